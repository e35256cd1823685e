// CUDA-core attention over [composed cache; suffix] with fp32 accumulation.
//
// This is the path for the fp32 context (no tensor-core format keeps fp32 inputs exact)
// and the fallback for shapes the tensor-core kernel does not take.  One CTA holds RB
// packed query rows of one (layer, request, KV head): row r = t * G + g is suffix token t,
// query head h_kv * G + g, so the G query heads that share a KV head reuse every K/V tile
// staged in shared memory.  Softmax is the streaming (online) form in base 2.
#include "internal.cuh"

#include <math_constants.h>

namespace c2kv {
namespace {

constexpr int RB = 16;    // query rows per CTA
constexpr int KT = 32;    // keys per staged tile (one per lane)
constexpr int NW = 4;     // warps per CTA
constexpr int RPW = RB / NW;

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

template <typename T, int D>
__global__ void __launch_bounds__(NW * 32) attn_simt_kernel(const __grid_constant__ AttnParams a) {
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

    for (int k0 = 0; k0 < nkeys; k0 += KT) {
        __syncthreads();
        for (int i = threadIdx.x; i < KT * D; i += NW * 32) {
            const int r = i / D, c = i - (i / D) * D;
            float kv = 0.f, vv = 0.f;
            if (k0 + r < nkeys) {
                kv = ldf(kb + (int64_t)(k0 + r) * row_stride + c);
                vv = ldf(vb + (int64_t)(k0 + r) * row_stride + c);
            }
            ks[r][c] = kv;
            vs[r][c] = vv;
        }
        __syncthreads();
#pragma unroll
        for (int rr = 0; rr < RPW; ++rr) {
            const int r = warp + NW * rr;
            const int pr = row0 + r;
            if (pr >= nrows) continue;          // warp-uniform
            const int t = pr / G;
            const int key = k0 + lane;
            float s = -CUDART_INF_F;
            if (key <= S + t && key < nkeys) {
                float dot = 0.f;
#pragma unroll 16
                for (int c = 0; c < D; ++c) dot = fmaf(qs[r][c], ks[lane][c], dot);
                s = dot * a.scale_log2;
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
#pragma unroll
            for (int c = 0; c < D / 32; ++c) acc[rr][c] *= alpha;
            for (int jk = 0; jk < KT; ++jk) {
                const float pj = __shfl_sync(0xffffffffu, p, jk);
#pragma unroll
                for (int c = 0; c < D / 32; ++c) acc[rr][c] = fmaf(pj, vs[jk][lane + 32 * c], acc[rr][c]);
            }
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
    if (dtype == kDtypeF32 && d == 64) return cudaFuncGetAttributes(&fa, attn_simt_kernel<float, 64>);
    if (dtype == kDtypeF32 && d == 128) return cudaFuncGetAttributes(&fa, attn_simt_kernel<float, 128>);
    if (dtype == kDtypeBf16 && d == 64) return cudaFuncGetAttributes(&fa, attn_simt_kernel<__nv_bfloat16, 64>);
    if (dtype == kDtypeBf16 && d == 128) return cudaFuncGetAttributes(&fa, attn_simt_kernel<__nv_bfloat16, 128>);
    return cudaErrorInvalidValue;
}

cudaError_t launch_attn_simt(const AttnParams& a, int dtype, int d, cudaStream_t s) {
    (void)cudaGetLastError();   // report this launch's error only, not a stale one
    const int G = a.hq / a.hkv;
    dim3 grid((a.sq * G + RB - 1) / RB, a.hkv, a.lq * a.batch);
    if (grid.z > 65535u) return cudaErrorInvalidValue;
    if (dtype == kDtypeF32 && d == 64) attn_simt_kernel<float, 64><<<grid, NW * 32, 0, s>>>(a);
    else if (dtype == kDtypeF32 && d == 128) attn_simt_kernel<float, 128><<<grid, NW * 32, 0, s>>>(a);
    else if (dtype == kDtypeBf16 && d == 64) attn_simt_kernel<__nv_bfloat16, 64><<<grid, NW * 32, 0, s>>>(a);
    else if (dtype == kDtypeBf16 && d == 128) attn_simt_kernel<__nv_bfloat16, 128><<<grid, NW * 32, 0, s>>>(a);
    else return cudaErrorInvalidValue;
    return cudaGetLastError();
}

}  // namespace c2kv
