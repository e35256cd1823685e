// CUDA-core attention over [composed cache; suffix] with fp32 accumulation.
//
// This is the path for the fp32 context (no tensor-core format keeps fp32 inputs exact)
// and the fallback for shapes the tensor-core kernel does not take.  One CTA holds RB
// packed query rows of one (layer, request, KV head): row r = t * G + g is suffix token t,
// query head h_kv * G + g, so the G query heads that share a KV head reuse every K/V tile
// staged in shared memory.  Softmax is the streaming (online) form in base 2.
//
// A small launch is bound by each warp's chain of dependent operations, not by bytes, so it
// takes RB = 4 (one row per warp, four times the CTAs) where RB = 16 would leave most SMs
// idle; the next K/V tile's loads are in flight while the current one is used; a score is
// four independent partial dot products, and P.V two.
#include "internal.cuh"

#include <math_constants.h>

namespace c2kv {
namespace {

constexpr int KT = 32;    // keys per staged tile (one per lane)
constexpr int NW = 4;     // warps per CTA

template <typename T>
__device__ __forceinline__ float ldf(const T* p);
template <>
__device__ __forceinline__ float ldf<float>(const float* p) { return __ldg(p); }
template <>
__device__ __forceinline__ float ldf<__nv_bfloat16>(const __nv_bfloat16* p) {
    return __bfloat162float(*p);
}
template <typename T>
__device__ __forceinline__ T stf(float x);
template <>
__device__ __forceinline__ float stf<float>(float x) { return x; }
template <>
__device__ __forceinline__ __nv_bfloat16 stf<__nv_bfloat16>(float x) {
    return __float2bfloat16_rn(x);
}

// RB query rows per CTA (RPW per warp).
template <typename T, int D, int RB>
__global__ void __launch_bounds__(NW * 32) attn_simt_kernel(const __grid_constant__ AttnParams a) {
    constexpr int RPW = RB / NW;
    static_assert(RPW * NW == RB, "rows per warp");
    __shared__ float qs[RB][D];
    __shared__ float ks[KT][D + 1];
    __shared__ float vs[KT][D];
    const int G = a.hq / a.hkv;
    const int l = blockIdx.z / a.batch;
    const int bl = blockIdx.z - l * a.batch;          // request within this launch
    const int b = a.b0 + bl;                          // request within the tensors
    const int hk = blockIdx.y;
    const int row0 = blockIdx.x * RB;
    const int nrows = a.sq * G;
    const T* q = static_cast<const T*>(a.q_rot);

    for (int i = threadIdx.x; i < RB * D; i += NW * 32) {
        const int r = i / D, c = i - (i / D) * D;
        const int pr = row0 + r;
        float val = 0.f;
        if (pr < nrows) {
            const int t = pr / G, g = pr - (pr / G) * G;
            const int64_t off = ((((int64_t)l * a.batch_total + b) * a.sq + t) * a.hq + hk * G + g) * D + c;
            val = ldf(q + off);
        }
        qs[r][c] = val;
    }

    const int S = a.req[bl].n_slots;
    const int64_t rb = a.req[bl].row_base;
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    float m[RPW], lsum[RPW], acc[RPW][D / 32];
#pragma unroll
    for (int rr = 0; rr < RPW; ++rr) {
        m[rr] = -CUDART_INF_F;
        lsum[rr] = 0.f;
#pragma unroll
        for (int c = 0; c < D / 32; ++c) acc[rr][c] = 0.f;
    }
    const int t_last = min(a.sq - 1, (row0 + RB - 1) / G);
    const int nkeys = S + t_last + 1;
    const int64_t row_stride = (int64_t)a.hkv * D;
    const T* kb = static_cast<const T*>(a.cache_k) +
                  (((int64_t)(a.layer0 + l) * a.rows + rb) * a.hkv + hk) * D;
    const T* vb = static_cast<const T*>(a.cache_v) +
                  (((int64_t)(a.layer0 + l) * a.rows + rb) * a.hkv + hk) * D;

    // this thread's share of a K/V tile, in registers until the tile before it is used
    constexpr int PER = KT * D / (NW * 32);
    static_assert(PER * NW * 32 == KT * D, "tile split over the threads");
    float kr[PER], vr[PER];
    auto fetch = [&](int k0) {
#pragma unroll
        for (int u = 0; u < PER; ++u) {
            const int i = (int)threadIdx.x + u * NW * 32;
            const int r = i / D, c = i - (i / D) * D;
            float kv = 0.f, vv = 0.f;
            if (k0 + r < nkeys) {
                kv = ldf(kb + (int64_t)(k0 + r) * row_stride + c);
                vv = ldf(vb + (int64_t)(k0 + r) * row_stride + c);
            }
            kr[u] = kv;
            vr[u] = vv;
        }
    };
    fetch(0);
    for (int k0 = 0; k0 < nkeys; k0 += KT) {
        __syncthreads();                      // the tile before this one is no longer read
#pragma unroll
        for (int u = 0; u < PER; ++u) {
            const int i = (int)threadIdx.x + u * NW * 32;
            const int r = i / D, c = i - (i / D) * D;
            ks[r][c] = kr[u];
            vs[r][c] = vr[u];
        }
        __syncthreads();
        if (k0 + KT < nkeys) fetch(k0 + KT);  // in flight while this tile is used
#pragma unroll
        for (int rr = 0; rr < RPW; ++rr) {
            const int r = warp + NW * rr;
            const int pr = row0 + r;
            if (pr >= nrows) continue;          // warp-uniform
            const int t = pr / G;
            const int key = k0 + lane;
            float s = -CUDART_INF_F;
            if (key <= S + t && key < nkeys) {
                float d0 = 0.f, d1 = 0.f, d2 = 0.f, d3 = 0.f;
#pragma unroll
                for (int c = 0; c < D; c += 4) {
                    d0 = fmaf(qs[r][c], ks[lane][c], d0);
                    d1 = fmaf(qs[r][c + 1], ks[lane][c + 1], d1);
                    d2 = fmaf(qs[r][c + 2], ks[lane][c + 2], d2);
                    d3 = fmaf(qs[r][c + 3], ks[lane][c + 3], d3);
                }
                s = ((d0 + d1) + (d2 + d3)) * a.scale_log2;
            }
            float mx = s;
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
            const float m_new = fmaxf(m[rr], mx);
            if (m_new == -CUDART_INF_F) continue;   // no visible key in this tile yet
            const float p = (s == -CUDART_INF_F) ? 0.f : exp2f(s - m_new);
            const float alpha = exp2f(m[rr] - m_new);
            float ps = p;
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) ps += __shfl_xor_sync(0xffffffffu, ps, o);
            lsum[rr] = lsum[rr] * alpha + ps;
            float pv0[D / 32], pv1[D / 32];      // P.V over the even and the odd keys
#pragma unroll
            for (int c = 0; c < D / 32; ++c) pv0[c] = pv1[c] = 0.f;
#pragma unroll
            for (int jk = 0; jk < KT; jk += 2) {
                const float pa = __shfl_sync(0xffffffffu, p, jk);
                const float pb = __shfl_sync(0xffffffffu, p, jk + 1);
#pragma unroll
                for (int c = 0; c < D / 32; ++c) {
                    pv0[c] = fmaf(pa, vs[jk][lane + 32 * c], pv0[c]);
                    pv1[c] = fmaf(pb, vs[jk + 1][lane + 32 * c], pv1[c]);
                }
            }
#pragma unroll
            for (int c = 0; c < D / 32; ++c) acc[rr][c] = fmaf(acc[rr][c], alpha, pv0[c] + pv1[c]);
            m[rr] = m_new;
        }
    }

    T* out = static_cast<T*>(a.out);
#pragma unroll
    for (int rr = 0; rr < RPW; ++rr) {
        const int pr = row0 + warp + NW * rr;
        if (pr >= nrows) continue;
        const int t = pr / G, g = pr - (pr / G) * G;
        const int h = hk * G + g;
        const float inv = 1.f / lsum[rr];
        const int64_t off = ((((int64_t)l * a.batch_total + b) * a.sq + t) * a.hq + h) * D;
#pragma unroll
        for (int c = 0; c < D / 32; ++c) out[off + lane + 32 * c] = stf<T>(acc[rr][c] * inv);
        if (a.lse != nullptr && lane == 0) {
            a.lse[(((int64_t)l * a.batch_total + b) * a.hq + h) * a.sq + t] =
                (m[rr] + log2f(lsum[rr])) * 0.69314718055994531f;
        }
    }
}

}  // namespace

cudaError_t preload_attn_simt_kernels(int dtype, int d) {
    cudaFuncAttributes fa{};
    cudaError_t e = cudaErrorInvalidValue;
    if (dtype == kDtypeF32 && d == 64) {
        e = cudaFuncGetAttributes(&fa, attn_simt_kernel<float, 64, 16>);
        if (e == cudaSuccess) e = cudaFuncGetAttributes(&fa, attn_simt_kernel<float, 64, 4>);
    } else if (dtype == kDtypeF32 && d == 128) {
        e = cudaFuncGetAttributes(&fa, attn_simt_kernel<float, 128, 16>);
        if (e == cudaSuccess) e = cudaFuncGetAttributes(&fa, attn_simt_kernel<float, 128, 4>);
    } else if (dtype == kDtypeBf16 && d == 64) {
        e = cudaFuncGetAttributes(&fa, attn_simt_kernel<__nv_bfloat16, 64, 16>);
        if (e == cudaSuccess) e = cudaFuncGetAttributes(&fa, attn_simt_kernel<__nv_bfloat16, 64, 4>);
    } else if (dtype == kDtypeBf16 && d == 128) {
        e = cudaFuncGetAttributes(&fa, attn_simt_kernel<__nv_bfloat16, 128, 16>);
        if (e == cudaSuccess) e = cudaFuncGetAttributes(&fa, attn_simt_kernel<__nv_bfloat16, 128, 4>);
    }
    return e;
}

namespace {
template <typename T, int D>
void launch_rb(const AttnParams& a, dim3 grid16, cudaStream_t s) {
    // 16 rows per CTA share each staged K/V tile; below two CTAs per SM of those (152 SMs)
    // the launch is latency-bound, and 4 rows per CTA spread it over four times the CTAs
    if ((int64_t)grid16.x * grid16.y * grid16.z < 2 * 152) {
        const int G = a.hq / a.hkv;
        const dim3 grid4((a.sq * G + 3) / 4, grid16.y, grid16.z);
        attn_simt_kernel<T, D, 4><<<grid4, NW * 32, 0, s>>>(a);
    } else {
        attn_simt_kernel<T, D, 16><<<grid16, NW * 32, 0, s>>>(a);
    }
}
}  // namespace

cudaError_t launch_attn_simt(const AttnParams& a, int dtype, int d, cudaStream_t s) {
    (void)cudaGetLastError();   // report this launch's error only, not a stale one
    const int G = a.hq / a.hkv;
    dim3 grid((a.sq * G + 15) / 16, a.hkv, a.lq * a.batch);
    if (grid.z > 65535u) return cudaErrorInvalidValue;
    if (dtype == kDtypeF32 && d == 64) launch_rb<float, 64>(a, grid, s);
    else if (dtype == kDtypeF32 && d == 128) launch_rb<float, 128>(a, grid, s);
    else if (dtype == kDtypeBf16 && d == 64) launch_rb<__nv_bfloat16, 64>(a, grid, s);
    else if (dtype == kDtypeBf16 && d == 128) launch_rb<__nv_bfloat16, 128>(a, grid, s);
    else return cudaErrorInvalidValue;
    return cudaGetLastError();
}

}  // namespace c2kv
