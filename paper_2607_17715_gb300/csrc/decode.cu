// Decode attention: one new token per request attends over its composed slots and the
// suffix rows written so far (the generation phase after the suffix, time between tokens).
//
// One query row per head and up to tens of thousands of keys: the work is reading K and V
// once (4 KB per key of a Llama-8B layer at bf16), so the kernel is HBM-bound and runs on
// the CUDA cores.  Each (layer, request, KV head) streams its key range split over several
// CTAs (flash-decoding).  In a CTA one producer lane streams 16 KB K and V tiles by TMA into
// a 3-stage shared-memory ring (two CTAs per SM keep 192 KB in flight, more than HBM latency
// needs at full bandwidth); four consumer warps keep the G query heads that share the KV head in
// registers, a group of LPK lanes covers one key row with one 16-byte shared-memory load per
// lane, and every lane group keeps its own online softmax (running max, sum and output
// slice).  The states of a CTA are merged in shared memory, and the CTAs of one row are
// merged by decode_merge_kernel with the exact log-sum-exp rule:
//     lse = log2 sum_s 2^lse_s,   O = sum_s 2^(lse_s - lse) O_s.
// Scores are kept in the log2 domain (the query is pre-scaled by log2(e) / sqrt(d)).
#include <math_constants.h>

#include <cstring>

#include "internal.cuh"
#include "ptx.cuh"
#include "vec16.cuh"

namespace c2kv {
namespace {


// (d0, d1) = (a0 b0 + c0, a1 b1 + c1) in one instruction (sm_100 packed f32x2; each lane is
// bitwise the scalar fmaf).
__device__ __forceinline__ void fma2(float& d0, float& d1, float a0, float a1, float b0, float b1,
                                     float c0, float c1) {
    asm("{\n\t.reg .b64 pa, pb, pc, pd;\n\t"
        "mov.b64 pa, {%2, %3};\n\t"
        "mov.b64 pb, {%4, %5};\n\t"
        "mov.b64 pc, {%6, %7};\n\t"
        "fma.rn.f32x2 pd, pa, pb, pc;\n\t"
        "mov.b64 {%0, %1}, pd;\n\t}"
        : "=f"(d0), "=f"(d1)
        : "f"(a0), "f"(a1), "f"(b0), "f"(b1), "f"(c0), "f"(c1));
}

__device__ __forceinline__ float ex2f(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

constexpr int kDecStages = 3;                    // ring depth
constexpr int kDecTileBytes = 16384;             // one K (or V) tile

struct DecodeTma {
    CUtensorMap tm_k;        // cache K [L*rows][Hkv][d], box {d, 1, KT}
    CUtensorMap tm_v;
    DecodeParams p;
};

constexpr size_t kDecSmem = 1024 + (size_t)kDecStages * 2 * kDecTileBytes + 16 * kDecStages + 16;

// Four consumer warps and the producer warp per CTA, two CTAs per SM: one CTA's start (the
// latency of its first tiles) overlaps the other's streaming.  For G >= 8 the query and
// output slices of a lane take too many registers for two CTAs, so one CTA runs eight
// consumer warps instead: two warps per SM sub-partition either way, so that one warp's
// chain of shuffles and dependent FMAs hides behind the other's.
template <int G>
__host__ __device__ constexpr int dec_consumers() { return G >= 8 ? 8 : 4; }
template <int G>
__host__ __device__ constexpr int dec_threads() { return (dec_consumers<G>() + 1) * 32; }

// T element type, D head dim, G query heads per KV head.
template <typename T, int D, int G>
__global__ void __launch_bounds__(dec_threads<G>(), G >= 8 ? 1 : 2) decode_kernel(const __grid_constant__ DecodeTma X) {
    const DecodeParams& P = X.p;
    constexpr int kDecConsumers = dec_consumers<G>();
    using V = Vec16<T>;
    constexpr int E = V::N;                            // elements per 16-byte vector
    constexpr int LPK = D / E;                         // lanes per key row
    constexpr int KPW = 32 / LPK;                      // key rows per warp pass
    constexpr int KT = kDecTileBytes / (D * (int)sizeof(T));   // keys per tile
    constexpr int KW = KT / kDecConsumers;             // keys of a tile per consumer warp
    constexpr int U_ALL = KW / KPW;                    // passes per warp per tile
    constexpr int U = U_ALL < 16 / G ? U_ALL : (16 / G > 0 ? 16 / G : 1);  // passes per round (U * G scores in registers)
    static_assert(LPK >= 1 && LPK <= 32 && 32 % LPK == 0, "lane mapping");
    static_assert(KW % KPW == 0 && U >= 1 && U_ALL % U == 0, "tile split over the consumer warps");

    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~uintptr_t(1023));
    const uint32_t sK = smem_u32(smem);
    const uint32_t sV = sK + kDecStages * kDecTileBytes;
    const uint32_t sBar = sV + kDecStages * kDecTileBytes;   // full[s], then empty[s]
    volatile uint32_t* abort = reinterpret_cast<volatile uint32_t*>(smem + 2 * kDecStages * kDecTileBytes +
                                                                   16 * kDecStages);
    auto full = [&](int st) { return sBar + 8u * (uint32_t)st; };
    auto empty = [&](int st) { return sBar + 8u * (uint32_t)(kDecStages + st); };

    __shared__ float sh_m[kDecConsumers][G];
    __shared__ float sh_l[kDecConsumers][G];
    __shared__ float sh_o[kDecConsumers][G][D];

    const int sp = blockIdx.x;
    const int hk = blockIdx.y;
    const int l = blockIdx.z / P.batch;
    const int bl = blockIdx.z - l * P.batch;
    const int b = P.b0 + bl;
    const ReqParam& rq = P.req[bl];
    const int n_keys = rq.n_slots + rq.t0 + 1;            // slots + suffix rows 0..step
    const int k_begin = sp * P.keys_per_split;
    const int k_end = min(n_keys, k_begin + P.keys_per_split);
    const int n_tiles = k_end > k_begin ? (k_end - k_begin + KT - 1) / KT : 0;

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int st = 0; st < kDecStages; ++st) {
            mbar_init(full(st), 1);
            mbar_init(empty(st), kDecConsumers);
        }
        *abort = 0u;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();

    if (warp == kDecConsumers) {
        // ---------------------------------------------------------------- TMA producer
        if (lane == 0 && n_tiles > 0) {
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&X.tm_k)) : "memory");
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&X.tm_v)) : "memory");
            const int row0 = (int)((int64_t)(P.layer0 + l) * P.rows + rq.row_base) + k_begin;
            for (int t = 0; t < n_tiles; ++t) {
                const int st = t % kDecStages;
                if (t >= kDecStages) mbar_wait(empty(st), (uint32_t)((t / kDecStages) - 1) & 1u, P.err, abort);
                // the step's own key row (the last key) is the suffix kernel's: every tile
                // before it is loaded while that kernel may still run
                if (t == n_tiles - 1 && k_end == n_keys) asm volatile("griddepcontrol.wait;" ::: "memory");
                mbar_expect_tx(full(st), 2 * kDecTileBytes);
                tma_load_3d(sK + st * kDecTileBytes, &X.tm_k, 0, hk, row0 + t * KT, full(st));
                tma_load_3d(sV + st * kDecTileBytes, &X.tm_v, 0, hk, row0 + t * KT, full(st));
            }
        }
        return;            // the producer takes no part in the merge below
    }

    // -------------------------------------------------------------------- consumers
    const int grp = lane / LPK;                           // key row slot within a pass
    const int c = lane - grp * LPK;                       // this lane's channels [cE, cE+E)
    const int64_t qrow = ((int64_t)l * P.batch_total + b) * P.hq + (int64_t)hk * G;
    asm volatile("griddepcontrol.wait;" ::: "memory");   // the rotated query is the suffix kernel's
    float q[G][E];
#pragma unroll
    for (int g = 0; g < G; ++g) {
        V::unpack(ld16(static_cast<const T*>(P.q_rot) + (qrow + g) * D + c * E), q[g]);
#pragma unroll
        for (int e = 0; e < E; ++e) q[g][e] *= P.scale_log2;
    }
    // The lane's own head after the reduce-scatter: bit k of it (from the top) is lane bit
    // LPK >> (k + 1).  mh, lh: that head's reference max and running sum; o: the output
    // slices of every head.
    constexpr int kLogG = G >= 16 ? 4 : G >= 8 ? 3 : G >= 4 ? 2 : G >= 2 ? 1 : 0;
    static_assert((1 << kLogG) == G && G <= LPK, "one head per lane after the reduce-scatter");
    const int gbase = lane & ~(LPK - 1);                  // first lane of this key row's group
    auto owner_off = [](int g) {                          // lane (within the group) owning head g
        int off = 0;
#pragma unroll
        for (int k = 0; k < kLogG; ++k)
            if ((g >> (kLogG - 1 - k)) & 1) off += LPK >> (k + 1);
        return off;
    };
    float mh = -CUDART_INF_F, lh = 0.f;
    float o[G][E];
#pragma unroll
    for (int g = 0; g < G; ++g)
#pragma unroll
        for (int e = 0; e < E; ++e) o[g][e] = 0.f;

    for (int t = 0; t < n_tiles; ++t) {                   // the same count for every warp
        const int st = t % kDecStages;
        mbar_wait(full(st), (uint32_t)(t / kDecStages) & 1u, P.err, abort);
        const uint8_t* kt = smem + (size_t)st * kDecTileBytes;
        const uint8_t* vt = smem + (size_t)(kDecStages + st) * kDecTileBytes;
#pragma unroll
        for (int u0 = 0; u0 < U_ALL; u0 += U) {
        const int key0 = k_begin + t * KT + warp * KW + u0 * KPW;   // first key of this round
        const int row0 = warp * KW + u0 * KPW;                       // its row within the tile
        float s[U][G];
        bool live[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int r = row0 + u * KPW + grp;           // row within the tile
            live[u] = key0 + u * KPW + grp < k_end;
            float kf[E];
            V::unpack(*reinterpret_cast<const uint4*>(kt + (size_t)r * D * sizeof(T) + c * 16), kf);
#pragma unroll
            for (int g = 0; g < G; ++g) {
                float a0 = 0.f, a1 = 0.f;                  // even and odd channels, packed
#pragma unroll
                for (int e = 0; e < E; e += 2) fma2(a0, a1, q[g][e], q[g][e + 1], kf[e], kf[e + 1], a0, a1);
                s[u][g] = a0 + a1;
            }
        }
        // Reduce-scatter the G partial dot products of each key row over its LPK lanes: at each
        // of the first log2(G) butterfly steps a lane keeps half of its heads and sends the
        // other half, so G - 1 exchanges leave every lane one full score, of head `hown`;
        // the remaining steps are plain sums (every lane of every consumer warp runs this:
        // the tile count is the same for all).
        float sr[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            float v[G];
#pragma unroll
            for (int g = 0; g < G; ++g) v[g] = s[u][g];
#pragma unroll
            for (int k = 0, nv = G; nv > 1; ++k, nv >>= 1) {
                const int off = LPK >> (k + 1);
                const bool hi = (lane & off) != 0;
#pragma unroll
                for (int i = 0; i < nv / 2; ++i) {
                    const float send = hi ? v[i] : v[i + nv / 2];
                    const float keep = hi ? v[i + nv / 2] : v[i];
                    v[i] = keep + __shfl_xor_sync(0xffffffffu, send, off);
                }
            }
#pragma unroll
            for (int off = LPK >> (kLogG + 1); off >= 1; off >>= 1)
                v[0] += __shfl_xor_sync(0xffffffffu, v[0], off);
            sr[u] = v[0];
        }
        // online softmax of the owned head against a reference max that moves only when the
        // head's max grows by more than 2^8 (the sum and the output use the same reference,
        // so the result is exact)
        float mx = -CUDART_INF_F;
#pragma unroll
        for (int u = 0; u < U; ++u)
            if (live[u]) mx = fmaxf(mx, sr[u]);
        const bool resc = mx > mh + 8.0f;                  // false while nothing is visible
        const float m_new = resc ? mx : mh;
        const float alpha = resc ? ex2f(mh - m_new) : 1.0f;  // 0 from -inf
        float pw[U];
        float psum = 0.f;
#pragma unroll
        for (int u = 0; u < U; ++u) {
            pw[u] = live[u] ? ex2f(sr[u] - m_new) : 0.f;
            psum += pw[u];
        }
        lh = lh * alpha + psum;
        mh = m_new;
        if (__any_sync(0xffffffffu, resc)) {              // rescale O for the heads that moved
#pragma unroll
            for (int g = 0; g < G; ++g) {
                const float a = __shfl_sync(0xffffffffu, alpha, gbase + owner_off(g));
#pragma unroll
                for (int e = 0; e < E; ++e) o[g][e] *= a;
            }
        }
        // every lane takes the weights of every head from their owners, then O += P V
        float pb[U][G];
#pragma unroll
        for (int u = 0; u < U; ++u)
#pragma unroll
            for (int g = 0; g < G; ++g) pb[u][g] = __shfl_sync(0xffffffffu, pw[u], gbase + owner_off(g));
#pragma unroll
        for (int u = 0; u < U; ++u) {
            if (!live[u]) continue;                        // rows past the range hold stale data
            const int r = row0 + u * KPW + grp;
            float vf[E];
            V::unpack(*reinterpret_cast<const uint4*>(vt + (size_t)r * D * sizeof(T) + c * 16), vf);
#pragma unroll
            for (int g = 0; g < G; ++g)
#pragma unroll
                for (int e = 0; e < E; e += 2)
                    fma2(o[g][e], o[g][e + 1], pb[u][g], pb[u][g], vf[e], vf[e + 1], o[g][e], o[g][e + 1]);
        }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(empty(st));             // this warp is done with the stage
    }

    // every head's (max, sum) from its owner to every lane of the key-row group
    float m[G], lsum[G];
#pragma unroll
    for (int g = 0; g < G; ++g) {
        m[g] = __shfl_sync(0xffffffffu, mh, gbase + owner_off(g));
        lsum[g] = __shfl_sync(0xffffffffu, lh, gbase + owner_off(g));
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
    // named barrier over the consumer warps only (the producer has left)
    asm volatile("bar.sync 1, %0;" ::"n"(kDecConsumers * 32) : "memory");
    // merge the warps: consumer thread i takes (head, channel) pairs i, i + 32 NC, ...
    for (int it = threadIdx.x; it < G * D; it += kDecConsumers * 32) {
        const int g = it / D;
        const int ch = it - g * D;
        float mm = -CUDART_INF_F;
#pragma unroll
        for (int w = 0; w < kDecConsumers; ++w) mm = fmaxf(mm, sh_m[w][g]);
        float ls = 0.f, os = 0.f;
        if (mm != -CUDART_INF_F) {
#pragma unroll
            for (int w = 0; w < kDecConsumers; ++w) {
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
// lane i owns channels i, i + 32, ...  The splits' lse values are fetched one per lane in a
// single round trip (up to 32 splits a round) and their maximum taken first, so the output
// slices that follow are independent loads.
template <typename T, int D>
__global__ void __launch_bounds__(256) decode_merge_kernel(const __grid_constant__ DecodeParams P) {
    const int64_t rows_all = (int64_t)P.lq * P.batch_total * P.hq;
    const int64_t row = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (row >= rows_all) return;                           // the whole warp leaves together
    // only the rows of this launch's requests
    const int64_t lb = row / P.hq;                         // l * Btot + b
    const int b = (int)(lb % P.batch_total);
    if (b < P.b0 || b >= P.b0 + P.batch) return;
    constexpr int PER = D / 32;
    float mm = -CUDART_INF_F;
    for (int s0 = 0; s0 < P.n_split; s0 += 32) {
        const int sl = s0 + lane;
        const float lse = sl < P.n_split ? P.part_lse[(int64_t)sl * rows_all + row] : -CUDART_INF_F;
        float m = lse;
#pragma unroll
        for (int off = 16; off >= 1; off >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, off));
        mm = fmaxf(mm, m);
    }
    float ls = 0.f;
    float acc[PER];
#pragma unroll
    for (int i = 0; i < PER; ++i) acc[i] = 0.f;
    if (mm != -CUDART_INF_F) {
#pragma unroll 4
        for (int s = 0; s < P.n_split; ++s) {
            const float lse = P.part_lse[(int64_t)s * rows_all + row];
            const float w = lse == -CUDART_INF_F ? 0.f : ex2f(lse - mm);
            const float* po = P.part_o + ((int64_t)s * rows_all + row) * D;
#pragma unroll
            for (int i = 0; i < PER; ++i) acc[i] = fmaf(w, po[lane + 32 * i], acc[i]);
            ls += w;
        }
    }
    const float inv = ls > 0.f ? 1.0f / ls : 0.f;
    T* dst = static_cast<T*>(P.out) + row * D;
#pragma unroll
    for (int i = 0; i < PER; ++i) dst[lane + 32 * i] = static_cast<T>(acc[i] * inv);
    if (lane == 0 && P.lse != nullptr) P.lse[row] = (mm + log2f(ls)) * 0.69314718055994531f;
}

template <typename T, int D, int G>
cudaError_t launch_g(const DecodeParams& p, cudaStream_t s, Hook before) {
    DecodeTma x;
    std::memset(&x, 0, sizeof(x));
    x.p = p;
    {   // K, V: cache [L*rows][Hkv][d] -> dims (d, Hkv, L*rows), one tile = KT whole rows
        constexpr int KT = kDecTileBytes / (D * (int)sizeof(T));
        const int64_t lrows = (int64_t)(p.layer0 + p.lq) * p.rows;
        const cuuint64_t dims[3] = {(cuuint64_t)D, (cuuint64_t)p.hkv, (cuuint64_t)lrows};
        const cuuint64_t str[2] = {(cuuint64_t)D * sizeof(T), (cuuint64_t)p.hkv * D * sizeof(T)};
        const cuuint32_t box[3] = {(cuuint32_t)D, 1, (cuuint32_t)KT};
        const CUtensorMapDataType ty =
            sizeof(T) == 2 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32;
        if (!encode_tensor_map(&x.tm_k, ty, 3, p.cache_k, dims, str, box, CU_TENSOR_MAP_SWIZZLE_NONE))
            return cudaErrorInvalidValue;
        if (!encode_tensor_map(&x.tm_v, ty, 3, p.cache_v, dims, str, box, CU_TENSOR_MAP_SWIZZLE_NONE))
            return cudaErrorInvalidValue;
    }
    // once per instantiation (a function-local static: thread-safe)
    static const cudaError_t smem_err = cudaFuncSetAttribute(
        decode_kernel<T, D, G>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kDecSmem);
    if (smem_err != cudaSuccess) return smem_err;
    cudaError_t e = cudaSuccess;
    const dim3 grid((unsigned)p.n_split, (unsigned)p.hkv, (unsigned)(p.lq * p.batch));
    before();
    if (p.dependent) {    // starts while the suffix kernel before it runs (see the waits above)
        cudaLaunchConfig_t cfg{};
        cfg.gridDim = grid;
        cfg.blockDim = dim3(dec_threads<G>());
        cfg.dynamicSmemBytes = kDecSmem;
        cfg.stream = s;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        e = cudaLaunchKernelEx(&cfg, decode_kernel<T, D, G>, x);
        if (e != cudaSuccess) return e;
    } else {
        decode_kernel<T, D, G><<<grid, dec_threads<G>(), kDecSmem, s>>>(x);
    }
    e = cudaGetLastError();
    if (e != cudaSuccess || p.n_split == 1) return e;
    const int64_t rows_all = (int64_t)p.lq * p.batch_total * p.hq;
    decode_merge_kernel<T, D><<<(unsigned)((rows_all + 7) / 8), 256, 0, s>>>(p);
    return cudaGetLastError();
}

template <typename T, int D>
cudaError_t launch_d(const DecodeParams& p, cudaStream_t s, Hook before) {
    switch (p.hq / p.hkv) {
        case 1: return launch_g<T, D, 1>(p, s, before);
        case 2: return launch_g<T, D, 2>(p, s, before);
        case 4: return launch_g<T, D, 4>(p, s, before);
        case 8: return launch_g<T, D, 8>(p, s, before);
        case 16:
            if constexpr (16 * D <= 1024 && 16 * Vec16<T>::N <= 64) return launch_g<T, D, 16>(p, s, before);
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

cudaError_t launch_decode(const DecodeParams& p, int dtype, cudaStream_t s, Hook before) {
    (void)cudaGetLastError();   // report this launch's error only, not a stale one
    if (p.batch < 1 || p.lq < 1) return cudaSuccess;
    if (p.n_split < 1 || (int64_t)p.lq * p.batch > 65535 || p.hkv > 65535) return cudaErrorInvalidValue;
    if (p.n_split > 1 && (p.part_o == nullptr || p.part_lse == nullptr)) return cudaErrorInvalidValue;
    if (dtype == kDtypeBf16)
        return p.d == 128 ? launch_d<__nv_bfloat16, 128>(p, s, before)
                          : p.d == 64 ? launch_d<__nv_bfloat16, 64>(p, s, before) : cudaErrorInvalidValue;
    return p.d == 128 ? launch_d<float, 128>(p, s, before)
                      : p.d == 64 ? launch_d<float, 64>(p, s, before) : cudaErrorInvalidValue;
}

}  // namespace c2kv
