// Extraction attention with the Structured Information Flow mask (Sec. 3.3): one attention
// layer of the C2 Extractor's forward over a chunk, given the Q, K, V of its n document
// tokens and m = ceil(n/k) C2 tokens (the trained projections that make them are the
// caller's).  The sequence is [x_0 .. x_{n-1}; c_0 .. c_{m-1}] with the C2 tokens grouped
// after the document (Sec. 3.3.1), and
//   * document token t sits at position t and sees document tokens 0..t only (original-token
//     invariance: its output is the frozen model's);
//   * C2 token c_j sits at the position of the last token of its block B(j) =
//     [jk, min((j+1)k, n)) and sees the document tokens of B(j) and of the sink block, and
//     the C2 tokens c_0 .. c_j (causal accumulation across blocks).
// The sink block B(0) of the paper's 1-based numbering is undefined by its block formula;
// it is read as the first block, [0, min(k, n)).
//
// extract_rope_kernel turns Q and K to those positions (fp32 arithmetic, stored in the
// context dtype like every cached activation).  The masked attention then takes one of two
// routes.
//
// Tensor cores (bf16, d = 128, the group sizes attn_tc_kernel takes).  The mask splits into
// pieces the suffix-attention kernel already computes:
//   1. document rows: plain causal attention over document keys 0..t, i.e. a "suffix" of n
//      tokens over an empty prefix;
//   2. C2 rows: a "suffix" of m tokens after n "slots", the document rows, so that c_j sees
//      c_0 .. c_j causally; the kernel's SIF mode (sif_k = k) masks every document key but
//      those of the sink block and B(j), and visits only the key tiles that hold them (for
//      a pair of 2 x 128 packed rows: its blocks' tiles, tile 0, the C2 tiles).
// Both are launches of attn_tc_kernel with a token pitch of n + m, so they read and write
// the extraction layout in place.
//
// CUDA cores (fp32, d = 64, other group sizes): extract_attn_kernel runs every row with fp32
// accumulation: one CTA holds RB packed query rows (row r = t * G + g: token t, query head
// h_kv * G + g) of one (layer, KV head), stages K/V tiles of KT keys in shared memory, and
// skips the tiles none of its rows can see.
#include <math_constants.h>

#include "internal.cuh"
#include "rope.cuh"
#include "vec16.cuh"

namespace c2kv {
namespace {

constexpr int XRB = 16;   // query rows per CTA
constexpr int XKT = 32;   // keys per staged tile (one per lane)
constexpr int XNW = 4;    // warps per CTA
constexpr int XRPW = XRB / XNW;

// Extraction position of token t of an (n, k) chunk.
__device__ __forceinline__ int extract_pos(int t, int n, int k) {
    if (t < n) return t;
    const int j = t - n;
    const int end = (j + 1) * k < n ? (j + 1) * k : n;
    return end - 1;
}

// Whether token tq may attend to token tk under the SIF mask.
__device__ __forceinline__ bool sif_visible(int tq, int tk, int n, int k) {
    if (tq < n) return tk <= tq;                               // document: causal, no C2 tokens
    const int j = tq - n;
    if (tk >= n) return tk - n <= j;                           // C2 tokens c_0 .. c_j
    const int blk = tk / k;
    return blk == j || blk == 0;                               // its block and the sink block
}

template <typename T, int VPH>
__global__ void __launch_bounds__(256) extract_rope_kernel(const __grid_constant__ ExtractParams P) {
    using V = Vec16<T>;
    constexpr int E = V::N;
    constexpr int HALF = VPH * E;
    constexpr int D = 2 * HALF;
    __shared__ float2 cs[HALF];
    const int t = blockIdx.x;
    const int l = blockIdx.y;
    const int pos = extract_pos(t, P.n, P.ratio);
    if (threadIdx.x < HALF) cs[threadIdx.x] = turn_cs(P.rope.turn[threadIdx.x], pos);
    __syncthreads();
    const int64_t row = (int64_t)l * P.n_all + t;               // token row of layer l
    const int nq = P.hq * VPH;
    const int items = (P.hq + P.hkv) * VPH;
    for (int p = threadIdx.x; p < items; p += blockDim.x) {
        const bool is_q = p < nq;
        const int pp = is_q ? p : p - nq;
        const int h = pp / VPH;
        const int iv = pp - h * VPH;
        const int heads = is_q ? P.hq : P.hkv;
        const int64_t off = (row * heads + h) * D + iv * E;
        const T* src = static_cast<const T*>(is_q ? P.q : P.k) + off;
        float x[E], y[E], gx[E], gy[E];
        V::unpack(ld16(src), x);
        V::unpack(ld16(src + HALF), y);
        rotate<E>(x, y, cs + iv * E, gx, gy);
        T* dst = static_cast<T*>(is_q ? P.q_rot : P.k_rot) + off;
        st16(dst, V::pack(gx));
        st16(dst + HALF, V::pack(gy));
    }
}

template <typename T>
__device__ __forceinline__ float ldx(const T* p) { return static_cast<float>(*p); }
template <>
__device__ __forceinline__ float ldx<__nv_bfloat16>(const __nv_bfloat16* p) { return __bfloat162float(*p); }

template <typename T, int D>
__global__ void __launch_bounds__(XNW * 32) extract_attn_kernel(const __grid_constant__ ExtractParams P) {
    __shared__ float qs[XRB][D];
    __shared__ float ks[XKT][D + 1];
    __shared__ float vs[XKT][D];
    const int G = P.hq / P.hkv;
    const int l = blockIdx.z;
    const int hk = blockIdx.y;
    const int row0 = blockIdx.x * XRB;
    const int nrows = P.n_all * G;
    const int n = P.n, k = P.ratio;
    const T* qr = static_cast<const T*>(P.q_rot);

    for (int i = threadIdx.x; i < XRB * D; i += XNW * 32) {
        const int r = i / D, c = i - (i / D) * D;
        const int pr = row0 + r;
        float val = 0.f;
        if (pr < nrows) {
            const int t = pr / G, g = pr - (pr / G) * G;
            val = ldx(qr + (((int64_t)l * P.n_all + t) * P.hq + hk * G + g) * D + c);
        }
        qs[r][c] = val;
    }

    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    float m[XRPW], lsum[XRPW], acc[XRPW][D / 32];
#pragma unroll
    for (int rr = 0; rr < XRPW; ++rr) {
        m[rr] = -CUDART_INF_F;
        lsum[rr] = 0.f;
#pragma unroll
        for (int c = 0; c < D / 32; ++c) acc[rr][c] = 0.f;
    }
    // key ranges some row of this CTA may see: causal document keys up to the last document
    // row, and for C2 rows c_ja .. c_jb the sink block, their blocks and c_0 .. c_jb
    const int tq0 = row0 / G;
    const int tq1 = min(P.n_all - 1, (row0 + XRB - 1) / G);
    const int doc_end = tq0 < n ? min(tq1, n - 1) + 1 : 0;
    const bool has_c2 = tq1 >= n;
    const int ja = max(tq0 - n, 0), jb = tq1 - n;
    const int sink_end = min(k, n);
    const int blk_lo = ja * k, blk_hi = has_c2 ? min((jb + 1) * k, n) : 0;
    const int c2_end = has_c2 ? n + jb + 1 : 0;
    auto tile_needed = [&](int k0) {
        const int k1 = k0 + XKT;
        if (k0 < doc_end) return true;
        if (!has_c2) return false;
        return k0 < sink_end || (k1 > blk_lo && k0 < blk_hi) || (k1 > n && k0 < c2_end);
    };
    const int nkeys = has_c2 ? c2_end : doc_end;
    const int64_t row_stride = (int64_t)P.hkv * D;
    const T* kb = static_cast<const T*>(P.k_rot) + ((int64_t)l * P.n_all * P.hkv + hk) * D;
    const T* vb = static_cast<const T*>(P.v) + ((int64_t)l * P.n_all * P.hkv + hk) * D;
    const float sc = P.scale_log2;

    for (int k0 = 0; k0 < nkeys; k0 += XKT) {
        if (!tile_needed(k0)) continue;                        // the same for the whole CTA
        __syncthreads();
        for (int i = threadIdx.x; i < XKT * D; i += XNW * 32) {
            const int r = i / D, c = i - (i / D) * D;
            float kv = 0.f, vv = 0.f;
            if (k0 + r < nkeys) {
                kv = ldx(kb + (int64_t)(k0 + r) * row_stride + c);
                vv = ldx(vb + (int64_t)(k0 + r) * row_stride + c);
            }
            ks[r][c] = kv;
            vs[r][c] = vv;
        }
        __syncthreads();
#pragma unroll
        for (int rr = 0; rr < XRPW; ++rr) {
            const int r = warp + XNW * rr;
            const int pr = row0 + r;
            if (pr >= nrows) continue;                           // warp-uniform
            const int tq = pr / G;
            const int tk = k0 + lane;
            float s = -CUDART_INF_F;
            if (tk < nkeys && sif_visible(tq, tk, n, k)) {
                float dot = 0.f;
#pragma unroll 16
                for (int c = 0; c < D; ++c) dot = fmaf(qs[r][c], ks[lane][c], dot);
                s = dot * sc;
            }
            float mx = s;
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
            const float m_new = fmaxf(m[rr], mx);
            if (m_new == -CUDART_INF_F) continue;                // warp-uniform: nothing visible yet
            const float p = (s == -CUDART_INF_F) ? 0.f : exp2f(s - m_new);
            const float alpha = exp2f(m[rr] - m_new);
            float ps = p;
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) ps += __shfl_xor_sync(0xffffffffu, ps, o);
            lsum[rr] = lsum[rr] * alpha + ps;
#pragma unroll
            for (int c = 0; c < D / 32; ++c) acc[rr][c] *= alpha;
            for (int jk = 0; jk < XKT; ++jk) {
                const float pj = __shfl_sync(0xffffffffu, p, jk);
#pragma unroll
                for (int c = 0; c < D / 32; ++c) acc[rr][c] = fmaf(pj, vs[jk][lane + 32 * c], acc[rr][c]);
            }
            m[rr] = m_new;
        }
    }

    T* out = static_cast<T*>(P.out);
#pragma unroll
    for (int rr = 0; rr < XRPW; ++rr) {
        const int pr = row0 + warp + XNW * rr;
        if (pr >= nrows) continue;
        const int t = pr / G, g = pr - (pr / G) * G;
        const int h = hk * G + g;
        const float inv = 1.f / lsum[rr];                        // every row sees itself
        const int64_t off = (((int64_t)l * P.n_all + t) * P.hq + h) * D;
#pragma unroll
        for (int c = 0; c < D / 32; ++c) out[off + lane + 32 * c] = static_cast<T>(acc[rr][c] * inv);
        if (P.lse != nullptr && lane == 0)
            P.lse[((int64_t)l * P.hq + h) * P.n_all + t] = (m[rr] + log2f(lsum[rr])) * 0.69314718055994531f;
    }
}

cudaError_t launch_tc(const ExtractParams& p, cudaStream_t s, cudaStream_t s2, cudaEvent_t fork,
                      cudaEvent_t join) {
    constexpr int D = 128;
    extract_rope_kernel<__nv_bfloat16, D / 2 / Vec16<__nv_bfloat16>::N>
        <<<dim3((unsigned)p.n_all, (unsigned)p.lq), 256, 0, s>>>(p);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    const int m = p.n_all - p.n;
    AttnParams a{};
    a.cache_k = p.k_rot;
    a.cache_v = p.v;
    a.err = p.err;
    a.rows = p.n_all;
    a.layer0 = 0;
    a.lq = p.lq;
    a.batch = 1;
    a.batch_total = 1;
    a.b0 = 0;
    a.sq_pitch = p.n_all;
    a.hq = p.hq;
    a.hkv = p.hkv;
    a.scale_log2 = p.scale_log2;
    a.n_split = 1;
    a.pairs_per_cta = p.pairs_per_cta;
    // piece 2 writes only the C2 rows (and reads the rotated rows): with a second stream it
    // runs beside piece 1, in the SMs its last wave of CTAs leaves idle
    cudaStream_t sc = s;
    if (s2 != nullptr) {
        e = cudaEventRecord(fork, s);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(s2, fork, 0);
        if (e != cudaSuccess) return e;
        sc = s2;
    }
    // 1. document rows over document keys 0..t
    a.q_rot = p.q_rot;
    a.out = p.out;
    a.lse = p.lse;
    a.sq = p.n;
    a.req[0] = ReqParam{0, 0, 0, 0};
    e = launch_attn_tc(a, s);
    if (e != cudaSuccess) return e;
    // 2. C2 rows: the n document rows as the request's slots, the C2 rows as its suffix, so
    // that c_j sees c_0 .. c_j causally; the kernel's SIF mode keeps, of the document keys,
    // the sink block and B(j), and visits only their key tiles
    const int64_t c2_off = (int64_t)p.n * p.hq * D;
    a.q_rot = static_cast<const __nv_bfloat16*>(p.q_rot) + c2_off;
    a.out = static_cast<__nv_bfloat16*>(p.out) + c2_off;
    a.lse = p.lse != nullptr ? p.lse + p.n : nullptr;
    a.sq = m;
    a.sif_k = p.ratio;
    a.req[0] = ReqParam{0, p.n, 0, 0};
    e = launch_attn_tc(a, sc);
    if (s2 != nullptr) {       // the work ends on s
        cudaError_t ej = cudaEventRecord(join, s2);
        if (ej == cudaSuccess) ej = cudaStreamWaitEvent(s, join, 0);
        if (e == cudaSuccess) e = ej;
    }
    return e;
}

template <typename T, int D>
cudaError_t launch_typed(const ExtractParams& p, cudaStream_t s) {
    constexpr int VPH = D / 2 / Vec16<T>::N;
    extract_rope_kernel<T, VPH><<<dim3((unsigned)p.n_all, (unsigned)p.lq), 256, 0, s>>>(p);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    const int G = p.hq / p.hkv;
    const dim3 grid((unsigned)((p.n_all * G + XRB - 1) / XRB), (unsigned)p.hkv, (unsigned)p.lq);
    extract_attn_kernel<T, D><<<grid, XNW * 32, 0, s>>>(p);
    return cudaGetLastError();
}

}  // namespace

bool extract_uses_tc(int dtype, int d, int hq, int hkv) { return attn_tc_supported(dtype, d, hq, hkv); }

cudaError_t launch_extract(const ExtractParams& p, int dtype, int d, cudaStream_t s, cudaStream_t s2,
                           cudaEvent_t fork, cudaEvent_t join) {
    (void)cudaGetLastError();   // report this launch's error only, not a stale one
    if (p.n_all < 1 || p.lq < 1) return cudaSuccess;
    if (p.lq > 65535 || p.hkv > 65535) return cudaErrorInvalidValue;
    if (extract_uses_tc(dtype, d, p.hq, p.hkv)) return launch_tc(p, s, s2, fork, join);
    if (dtype == kDtypeF32 && d == 64) return launch_typed<float, 64>(p, s);
    if (dtype == kDtypeF32 && d == 128) return launch_typed<float, 128>(p, s);
    if (dtype == kDtypeBf16 && d == 64) return launch_typed<__nv_bfloat16, 64>(p, s);
    if (dtype == kDtypeBf16 && d == 128) return launch_typed<__nv_bfloat16, 128>(p, s);
    return cudaErrorInvalidValue;
}

}  // namespace c2kv
