// Decode attention: one new token per request attends over its composed slots and the
// suffix rows written so far (the generation phase after the suffix, time between tokens).
//
// One query row per head and up to tens of thousands of keys: the work is reading K and V
// once (4 KB per key of a Llama-8B layer at bf16), so the kernel is HBM-bound and runs on
// the CUDA cores.  Each (layer, request, KV head) streams its key range split over several
// CTAs (flash-decoding): a CTA keeps the G query heads that share the KV head in registers,
// a group of LPK lanes covers one key row with one 16-byte load per lane, and every lane
// group keeps its own online softmax (running max, sum and output slice).  The states of a
// CTA are merged in shared memory, and the CTAs of one row are merged by
// decode_merge_kernel with the exact log-sum-exp rule:
//     lse = log2 sum_s 2^lse_s,   O = sum_s 2^(lse_s - lse) O_s.
// Scores are kept in the log2 domain (the query is pre-scaled by log2(e) / sqrt(d)).
#include <math_constants.h>

#include "internal.cuh"
#include "vec16.cuh"

namespace c2kv {
namespace {

constexpr int kDecThreads = 256;
constexpr int kDecWarps = kDecThreads / 32;

__device__ __forceinline__ float ex2f(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// T element type, D head dim, G query heads per KV head, U keys in flight per lane group.
template <typename T, int D, int G, int U>
__global__ void __launch_bounds__(kDecThreads, G <= 4 ? 2 : 1) decode_kernel(const __grid_constant__ DecodeParams P) {
    using V = Vec16<T>;
    constexpr int E = V::N;            // elements per 16-byte vector
    constexpr int LPK = D / E;         // lanes per key row
    constexpr int KPW = 32 / LPK;      // key rows per warp step
    constexpr int STEP = KPW * kDecWarps;
    static_assert(LPK >= 1 && LPK <= 32 && 32 % LPK == 0, "lane mapping");

    __shared__ float sh_m[kDecWarps][G];
    __shared__ float sh_l[kDecWarps][G];
    __shared__ float sh_o[kDecWarps][G][D];

    const int sp = blockIdx.x;
    const int hk = blockIdx.y;
    const int l = blockIdx.z / P.batch;
    const int bl = blockIdx.z - l * P.batch;
    const int b = P.b0 + bl;
    const ReqParam& rq = P.req[bl];
    const int n_keys = rq.n_slots + rq.t0 + 1;            // slots + suffix rows 0..step
    const int k_begin = sp * P.keys_per_split;
    const int k_end = min(n_keys, k_begin + P.keys_per_split);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int grp = lane / LPK;                           // key row slot within the warp
    const int c = lane - grp * LPK;                       // this lane's channels [cE, cE+E)
    const int64_t row_elems = (int64_t)P.hkv * D;
    const int64_t qrow = ((int64_t)l * P.batch_total + b) * P.hq + (int64_t)hk * G;

    float q[G][E];
#pragma unroll
    for (int g = 0; g < G; ++g) {
        V::unpack(ld16(static_cast<const T*>(P.q_rot) + (qrow + g) * D + c * E), q[g]);
#pragma unroll
        for (int e = 0; e < E; ++e) q[g][e] *= P.scale_log2;
    }
    float m[G], lsum[G], o[G][E];
#pragma unroll
    for (int g = 0; g < G; ++g) {
        m[g] = -CUDART_INF_F;
        lsum[g] = 0.f;
#pragma unroll
        for (int e = 0; e < E; ++e) o[g][e] = 0.f;
    }

    const T* kbase = static_cast<const T*>(P.cache_k) +
                     ((int64_t)(P.layer0 + l) * P.rows + rq.row_base) * row_elems + (int64_t)hk * D + c * E;
    const T* vbase = static_cast<const T*>(P.cache_v) +
                     ((int64_t)(P.layer0 + l) * P.rows + rq.row_base) * row_elems + (int64_t)hk * D + c * E;

    // The loop bound is the warp's first key, the same for every lane: the shuffles below
    // take the full warp, so no lane group may leave the loop before the others (a key past
    // the range is masked instead).
    for (int kw = k_begin + warp * KPW; kw < k_end; kw += U * STEP) {
        const int k0 = kw + grp;
        uint4 kr[U], vr[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {                     // every load of the step in flight
            const int key = k0 + u * STEP;
            if (key < k_end) {
                kr[u] = ld16(kbase + (int64_t)key * row_elems);
                vr[u] = ld16(vbase + (int64_t)key * row_elems);
            } else {
                kr[u] = make_uint4(0, 0, 0, 0);
                vr[u] = kr[u];
            }
        }
        float s[U][G];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            float kf[E];
            V::unpack(kr[u], kf);
#pragma unroll
            for (int g = 0; g < G; ++g) {
                float acc = 0.f;
#pragma unroll
                for (int e = 0; e < E; ++e) acc = fmaf(q[g][e], kf[e], acc);
                s[u][g] = acc;
            }
        }
        // reduce the partial dot products over the LPK lanes of each key row
#pragma unroll
        for (int off = LPK / 2; off >= 1; off >>= 1)
#pragma unroll
            for (int u = 0; u < U; ++u)
#pragma unroll
                for (int g = 0; g < G; ++g) s[u][g] += __shfl_xor_sync(0xffffffffu, s[u][g], off);
#pragma unroll
        for (int g = 0; g < G; ++g) {
            float mx = m[g];
#pragma unroll
            for (int u = 0; u < U; ++u)
                if (k0 + u * STEP < k_end) mx = fmaxf(mx, s[u][g]);
            const float alpha = ex2f(m[g] - mx);           // 0 while m = -inf
            lsum[g] *= alpha;
#pragma unroll
            for (int e = 0; e < E; ++e) o[g][e] *= alpha;
            m[g] = mx;
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const bool live = k0 + u * STEP < k_end;
            float vf[E];
            V::unpack(vr[u], vf);
#pragma unroll
            for (int g = 0; g < G; ++g) {
                const float p = live ? ex2f(s[u][g] - m[g]) : 0.f;
                lsum[g] += p;
#pragma unroll
                for (int e = 0; e < E; ++e) o[g][e] = fmaf(p, vf[e], o[g][e]);
            }
        }
    }

    // merge the lane groups of a warp (lanes c, c + LPK, ... hold the same channels)
#pragma unroll
    for (int off = LPK; off < 32; off <<= 1) {
#pragma unroll
        for (int g = 0; g < G; ++g) {
            const float m2 = __shfl_xor_sync(0xffffffffu, m[g], off);
            const float l2 = __shfl_xor_sync(0xffffffffu, lsum[g], off);
            const float mm = fmaxf(m[g], m2);
            const float a1 = mm == -CUDART_INF_F ? 0.f : ex2f(m[g] - mm);
            const float a2 = mm == -CUDART_INF_F ? 0.f : ex2f(m2 - mm);
#pragma unroll
            for (int e = 0; e < E; ++e) {
                const float o2 = __shfl_xor_sync(0xffffffffu, o[g][e], off);
                o[g][e] = o[g][e] * a1 + o2 * a2;
            }
            lsum[g] = lsum[g] * a1 + l2 * a2;
            m[g] = mm;
        }
    }
    if (grp == 0) {
#pragma unroll
        for (int g = 0; g < G; ++g) {
            if (c == 0) {
                sh_m[warp][g] = m[g];
                sh_l[warp][g] = lsum[g];
            }
#pragma unroll
            for (int e = 0; e < E; ++e) sh_o[warp][g][c * E + e] = o[g][e];
        }
    }
    __syncthreads();
    // merge the warps: thread i takes (head, channel) pairs i, i + 256, ...
    for (int it = threadIdx.x; it < G * D; it += kDecThreads) {
        const int g = it / D;
        const int ch = it - g * D;
        float mm = -CUDART_INF_F;
#pragma unroll
        for (int w = 0; w < kDecWarps; ++w) mm = fmaxf(mm, sh_m[w][g]);
        float ls = 0.f, os = 0.f;
        if (mm != -CUDART_INF_F) {
#pragma unroll
            for (int w = 0; w < kDecWarps; ++w) {
                const float a = ex2f(sh_m[w][g] - mm);
                ls += sh_l[w][g] * a;
                os += sh_o[w][g][ch] * a;
            }
        }
        const int64_t row = qrow + g;                      // (l * Btot + b) * Hq + h
        const float inv = ls > 0.f ? 1.0f / ls : 0.f;
        if (P.n_split == 1) {
            T* dst = static_cast<T*>(P.out) + row * D + ch;
            *dst = static_cast<T>(os * inv);
            if (ch == 0 && P.lse != nullptr) P.lse[row] = (mm + log2f(ls)) * 0.69314718055994531f;
        } else {
            const int64_t rows_all = (int64_t)P.lq * P.batch_total * P.hq;
            P.part_o[((int64_t)sp * rows_all + row) * D + ch] = os * inv;
            if (ch == 0) P.part_lse[(int64_t)sp * rows_all + row] = ls > 0.f ? mm + log2f(ls) : -CUDART_INF_F;
        }
    }
}

// Merge the key-range splits of each (layer, request, query head) row.  One warp per row;
// lane i owns channels i, i + 32, ...
template <typename T, int D>
__global__ void __launch_bounds__(256) decode_merge_kernel(const __grid_constant__ DecodeParams P) {
    const int64_t rows_all = (int64_t)P.lq * P.batch_total * P.hq;
    const int64_t row = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (row >= rows_all) return;
    // only the rows of this launch's requests
    const int64_t lb = row / P.hq;                         // l * Btot + b
    const int b = (int)(lb % P.batch_total);
    if (b < P.b0 || b >= P.b0 + P.batch) return;
    constexpr int PER = D / 32;
    float mm = -CUDART_INF_F, ls = 0.f;
    float acc[PER];
#pragma unroll
    for (int i = 0; i < PER; ++i) acc[i] = 0.f;
    for (int s = 0; s < P.n_split; ++s) {
        const float lse = P.part_lse[(int64_t)s * rows_all + row];
        if (lse == -CUDART_INF_F) continue;                // no key in this split
        const float m2 = fmaxf(mm, lse);
        const float a = ex2f(mm - m2);                     // 0 while mm = -inf
        const float w = ex2f(lse - m2);
        const float* po = P.part_o + ((int64_t)s * rows_all + row) * D;
#pragma unroll
        for (int i = 0; i < PER; ++i) acc[i] = acc[i] * a + w * po[lane + 32 * i];
        ls = ls * a + w;
        mm = m2;
    }
    const float inv = ls > 0.f ? 1.0f / ls : 0.f;
    T* dst = static_cast<T*>(P.out) + row * D;
#pragma unroll
    for (int i = 0; i < PER; ++i) dst[lane + 32 * i] = static_cast<T>(acc[i] * inv);
    if (lane == 0 && P.lse != nullptr) P.lse[row] = (mm + log2f(ls)) * 0.69314718055994531f;
}

template <typename T, int D, int G>
cudaError_t launch_g(const DecodeParams& p, cudaStream_t s) {
    // keys in flight per lane group: as many as the registers of two CTAs per SM allow
    constexpr int GE = G * Vec16<T>::N;
    constexpr int U = GE <= 16 ? 4 : GE <= 32 ? 3 : 2;
    const dim3 grid((unsigned)p.n_split, (unsigned)p.hkv, (unsigned)(p.lq * p.batch));
    decode_kernel<T, D, G, U><<<grid, kDecThreads, 0, s>>>(p);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess || p.n_split == 1) return e;
    const int64_t rows_all = (int64_t)p.lq * p.batch_total * p.hq;
    decode_merge_kernel<T, D><<<(unsigned)((rows_all + 7) / 8), 256, 0, s>>>(p);
    return cudaGetLastError();
}

template <typename T, int D>
cudaError_t launch_d(const DecodeParams& p, cudaStream_t s) {
    switch (p.hq / p.hkv) {
        case 1: return launch_g<T, D, 1>(p, s);
        case 2: return launch_g<T, D, 2>(p, s);
        case 4: return launch_g<T, D, 4>(p, s);
        case 8: return launch_g<T, D, 8>(p, s);
        case 16:
            if constexpr (16 * D <= 1024 && 16 * Vec16<T>::N <= 64) return launch_g<T, D, 16>(p, s);
            return cudaErrorInvalidValue;
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace

bool decode_supported(int dtype, int d, int hq, int hkv) {
    if (hkv < 1 || hq % hkv) return false;
    const int g = hq / hkv;
    if (g != 1 && g != 2 && g != 4 && g != 8 && g != 16) return false;
    if (dtype != kDtypeBf16 && dtype != kDtypeF32) return false;
    const int e = dtype == kDtypeBf16 ? 8 : 4;        // elements per 16-byte vector
    // per-warp partials fit shared memory; query and output slices fit registers
    return (d == 64 || d == 128) && g * d <= 1024 && g * e <= 64;
}

cudaError_t launch_decode(const DecodeParams& p, int dtype, cudaStream_t s) {
    (void)cudaGetLastError();   // report this launch's error only, not a stale one
    if (p.batch < 1 || p.lq < 1) return cudaSuccess;
    if (p.n_split < 1 || (int64_t)p.lq * p.batch > 65535 || p.hkv > 65535) return cudaErrorInvalidValue;
    if (p.n_split > 1 && (p.part_o == nullptr || p.part_lse == nullptr)) return cudaErrorInvalidValue;
    if (dtype == kDtypeBf16)
        return p.d == 128 ? launch_d<__nv_bfloat16, 128>(p, s) : p.d == 64 ? launch_d<__nv_bfloat16, 64>(p, s)
                                                                          : cudaErrorInvalidValue;
    return p.d == 128 ? launch_d<float, 128>(p, s) : p.d == 64 ? launch_d<float, 64>(p, s) : cudaErrorInvalidValue;
}

}  // namespace c2kv
