// Streaming KV kernels of the C2KV hot path: compose (re-rotate + gather), compress (block
// mean + local RoPE), suffix preparation.  All are HBM-bound element-wise moves: each
// thread moves 16-byte vectors, and one thread owns a RoPE pair of vectors (channels
// [c, c+E) and [c + d/2, c + d/2 + E)) so the 2x2 rotation needs no exchange between
// threads.
//
// Angles: cos/sin of p * theta^(-2i/d) come from the phase accumulator in RopeTurns (the
// turn fraction is the low 64 bits of p * turn[i], exact integer wrap-around), converted
// once to a float in [-1/2, 1/2) turns and handed to sincospif.  The error is about
// 1e-7 rad at any position, where forming p * inv_freq in fp32 would lose p * 2^-24 rad.
#include <algorithm>

#include "internal.cuh"
#include "rope.cuh"
#include "vec16.cuh"

namespace c2kv {
namespace {


// (cos, sin) of pos * theta^(-2i/d) from the 0.64 fixed-point turn of frequency i.

// ---------------------------------------------------------------------------------------
// compose.  grid = (CTAs per layer, layers); a tile is P.tile_slots (<= kComposeTile)
// consecutive slots of one chunk occurrence, and CTA x takes tiles x, x + gridDim.x, ...
// (one each unless the launch caps its CTAs).  Per tile the CTA forms the d/2 (cos, sin) of
// the turn in shared memory -- once for the occurrence's offset delta (LOCAL_ROPE storage),
// or per slot for its composed position delta + p_j (PRE_ROPE storage, K stored before
// RoPE) -- then streams the tile: per item (slot, head, vector pair) four 16-byte loads of
// stored K/V, K turned, four 16-byte stores into the composed cache.  IPT items per thread
// are loaded before any is stored, so 16 loads per thread are in flight.  The launch sizes
// the CTA to the tile (tile items / IPT threads, 32 to 256), so a launch of small tiles
// keeps every thread's loads in flight and spreads evenly over the SMs.
// ---------------------------------------------------------------------------------------
template <typename T, int VPH>
__global__ void __launch_bounds__(256) compose_kernel(const __grid_constant__ ComposeParams P) {
    using V = Vec16<T>;
    constexpr int E = V::N;
    constexpr int HALF = VPH * E;
    constexpr int D = 2 * HALF;
    constexpr int IPT = 4;
    __shared__ float2 cs[kComposeTile * HALF];
    const int l = P.layer0 + (int)blockIdx.y;
    const int ts = P.tile_slots;
    for (int tile = blockIdx.x; tile < P.n_tiles; tile += gridDim.x) {
        int lo = 0, hi = P.n_occ - 1;
        while (lo < hi) {                       // last occurrence whose tile_base <= tile
            const int mid = (lo + hi + 1) >> 1;
            if (P.occ[mid].tile_base <= tile) lo = mid;
            else hi = mid - 1;
        }
        const OccParam& o = P.occ[lo];
        const int j0 = (tile - o.tile_base) * ts;
        const int ns = min(ts, o.m - j0);
        __syncthreads();                        // the previous tile is done with cs
        if (!P.pre_rope) {
            for (int i = threadIdx.x; i < HALF; i += blockDim.x) cs[i] = turn_cs(P.rope.turn[i], o.delta);
        } else {
            // row s of the table: slot j0 + s at its composed position delta + p_j
            for (int e = threadIdx.x; e < ns * HALF; e += blockDim.x) {
                const int s = e / HALF, i = e - s * HALF;
                const int64_t pos = (int64_t)o.delta + min((j0 + s + 1) * o.k, o.n) - 1;
                cs[e] = turn_cs(P.rope.turn[i], pos);
            }
        }
        __syncthreads();
        if (ns <= 0) continue;                  // the same for the whole CTA

        const T* __restrict__ pk = static_cast<const T*>(P.pool_k);
        const T* __restrict__ pv = static_cast<const T*>(P.pool_v);
        T* __restrict__ ok = static_cast<T*>(P.out_k);
        T* __restrict__ ov = static_cast<T*>(P.out_v);
        const int pairs = P.hkv * VPH;
        const int items = ns * pairs;
        const int64_t row_elems = (int64_t)P.hkv * D;

        const int nthr = (int)blockDim.x;
        for (int base = 0; base < items; base += nthr * IPT) {
            uint4 kx[IPT], ky[IPT], vx[IPT], vy[IPT];
            int64_t dof[IPT];
            int civ[IPT];
            bool live[IPT];
    #pragma unroll
            for (int u = 0; u < IPT; ++u) {
                const int it = base + u * nthr + (int)threadIdx.x;
                live[u] = it < items;
                if (!live[u]) continue;
                const int s = it / pairs;
                const int p = it - s * pairs;
                const int h = p / VPH;
                const int iv = p - h * VPH;
                const int j = j0 + s;
                const int64_t src = (int64_t)o.src_base + j;
                const int64_t dst = (int64_t)o.dest_row + j;
                if ((!o.host && (src < 0 || src >= P.pool_slots)) || dst < 0 || dst >= P.rows) {
                    atomicOr(P.err, 1);
                    live[u] = false;
                    continue;
                }
                dof[u] = ((int64_t)l * P.rows + dst) * row_elems + h * D + iv * E;
                civ[u] = (P.pre_rope ? s * HALF : 0) + iv * E;
                const T* sk;
                const T* sv;
                if (o.host) {       // host-resident chunk: [L][m][Hkv][d] read over the host link
                    const int64_t so = ((int64_t)l * o.m + j) * row_elems + h * D + iv * E;
                    sk = static_cast<const T*>(o.host_k) + so;
                    sv = static_cast<const T*>(o.host_v) + so;
                } else {
                    const int64_t so = ((int64_t)l * P.pool_slots + src) * row_elems + h * D + iv * E;
                    sk = pk + so;
                    sv = pv + so;
                }
                kx[u] = ld16(sk);
                ky[u] = ld16(sk + HALF);
                vx[u] = ld16(sv);
                vy[u] = ld16(sv + HALF);
                if (l == 0 && p == 0) P.pos[dst] = o.delta + min((j + 1) * o.k, o.n) - 1;
            }
    #pragma unroll
            for (int u = 0; u < IPT; ++u) {
                if (!live[u]) continue;
                float fx[E], fy[E], gx[E], gy[E];
                V::unpack(kx[u], fx);
                V::unpack(ky[u], fy);
                rotate<E>(fx, fy, cs + civ[u], gx, gy);
                st16(ok + dof[u], V::pack(gx));
                st16(ok + dof[u] + HALF, V::pack(gy));
                st16(ov + dof[u], vx[u]);
                st16(ov + dof[u] + HALF, vy[u]);
            }
        }
    }
}

// ---------------------------------------------------------------------------------------
// compress: one item = (layer, slot, head, vector pair).  Mean of the block's rows (or the
// provided slot row), K turned to the slot's local position (LOCAL_ROPE storage; kept as is
// under PRE_ROPE), both stored in the pool.
// ---------------------------------------------------------------------------------------
template <typename T, int VPH>
__global__ void __launch_bounds__(256) compress_kernel(const __grid_constant__ CompressParams P) {
    using V = Vec16<T>;
    constexpr int E = V::N;
    constexpr int HALF = VPH * E;
    constexpr int D = 2 * HALF;
    const int pairs = P.hkv * VPH;
    const int64_t per_layer = (int64_t)P.m * pairs;
    const int64_t total = per_layer * P.layers;
    const int64_t row_elems = (int64_t)P.hkv * D;
    const T* ik = static_cast<const T*>(P.in_k);
    const T* iv_ = static_cast<const T*>(P.in_v);
    T* pk = static_cast<T*>(P.pool_k);
    T* pv = static_cast<T*>(P.pool_v);
    for (int64_t it = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; it < total;
         it += (int64_t)gridDim.x * blockDim.x) {
        const int l = (int)(it / per_layer);
        const int64_t r = it - (int64_t)l * per_layer;
        const int j = (int)(r / pairs);
        const int p = (int)(r - (int64_t)j * pairs);
        const int h = p / VPH;
        const int iv = p - h * VPH;
        int r0, r1;
        if (P.one_row) {
            r0 = j;
            r1 = j + 1;
        } else {
            r0 = j * P.k;
            r1 = min(r0 + P.k, P.n);
        }
        float sx[E], sy[E], tx[E], ty[E];
#pragma unroll
        for (int e = 0; e < E; ++e) sx[e] = sy[e] = tx[e] = ty[e] = 0.f;
        for (int row = r0; row < r1; ++row) {
            const int64_t off = ((int64_t)l * P.rows_in + row) * row_elems + h * D + iv * E;
            float f[E];
            V::unpack(ld16(ik + off), f);
#pragma unroll
            for (int e = 0; e < E; ++e) sx[e] += f[e];
            V::unpack(ld16(ik + off + HALF), f);
#pragma unroll
            for (int e = 0; e < E; ++e) sy[e] += f[e];
            V::unpack(ld16(iv_ + off), f);
#pragma unroll
            for (int e = 0; e < E; ++e) tx[e] += f[e];
            V::unpack(ld16(iv_ + off + HALF), f);
#pragma unroll
            for (int e = 0; e < E; ++e) ty[e] += f[e];
        }
        const int cnt = r1 - r0;
        if (cnt > 1) {
            const float c = (float)cnt;
#pragma unroll
            for (int e = 0; e < E; ++e) {
                sx[e] = sx[e] / c;
                sy[e] = sy[e] / c;
                tx[e] = tx[e] / c;
                ty[e] = ty[e] / c;
            }
        }
        // slot j sits at the last token of its block (provided slots: same rule)
        const int64_t p_local = (int64_t)min((j + 1) * P.k, P.n) - 1;
        float gx[E], gy[E];
        if (P.turn) {
            float2 cs[E];
#pragma unroll
            for (int e = 0; e < E; ++e) cs[e] = turn_cs(P.rope.turn[iv * E + e], p_local);
            rotate<E>(sx, sy, cs, gx, gy);
        } else {            // PRE_ROPE storage: the slot's K before any positional embedding
#pragma unroll
            for (int e = 0; e < E; ++e) {
                gx[e] = sx[e];
                gy[e] = sy[e];
            }
        }
        const int64_t dof =
            ((int64_t)l * P.pool_slots + P.slot_base + j) * row_elems + h * D + iv * E;
        st16(pk + dof, V::pack(gx));
        st16(pk + dof + HALF, V::pack(gy));
        st16(pv + dof, V::pack(tx));
        st16(pv + dof + HALF, V::pack(ty));
    }
}

// ---------------------------------------------------------------------------------------
// suffix preparation.  grid = (batch * kPadParts pad blocks + batch * Sq suffix rows,
// layers).  A pad block zeroes every kPadParts-th cache row of its request from the end of
// the suffix to the next 128-row boundary, so a key tile that straddles the end reads finite
// zeros (masked keys must not carry NaN/Inf garbage into P.V); the pad blocks come first in
// the grid and share the work, so that none trails the launch.  A row block issues its
// loads of the row's Hq query heads and Hkv key/value heads first, forms the row's d/2
// (cos, sin) at L_b + t in shared memory while they are in flight, then turns the queries
// into q_rot and the keys into the cache row row_base + S_b + t (V copied alongside).
// ---------------------------------------------------------------------------------------
constexpr int kPadParts = 4;

template <typename T, int VPH>
__global__ void __launch_bounds__(256) suffix_kernel(const __grid_constant__ SuffixParams P) {
    using V = Vec16<T>;
    constexpr int E = V::N;
    constexpr int HALF = VPH * E;
    constexpr int D = 2 * HALF;
    // a programmatic dependent (the decode kernel) may start now: it waits
    // (griddepcontrol.wait) before it reads what this kernel writes
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    __shared__ float2 cs[HALF];
    const int l = blockIdx.y;
    const int n_pad = P.pad_rows ? P.batch * kPadParts : 0;
    const int64_t row_elems = (int64_t)P.hkv * D;
    if ((int)blockIdx.x < n_pad) {
        const int bl = (int)blockIdx.x / kPadParts;
        const int part = (int)blockIdx.x - bl * kPadParts;
        const int used = P.pad_from[bl];
        const int end = (used + 127) / 128 * 128;
        constexpr int VPR_ELEMS = 16 / (int)sizeof(T);
        const int vec_per_row = (int)(row_elems / VPR_ELEMS);
        const int rows = end - used > part ? (end - used - part + kPadParts - 1) / kPadParts : 0;
        const int items = rows * vec_per_row;
        const uint4 z = make_uint4(0, 0, 0, 0);
        for (int it = threadIdx.x; it < items; it += blockDim.x) {
            const int rr = it / vec_per_row;
            const int vi = it - rr * vec_per_row;
            const int64_t crow = (int64_t)P.req[bl].row_base + used + part + (int64_t)rr * kPadParts;
            if (crow >= P.rows) continue;
            const int64_t off = ((int64_t)(P.layer0 + l) * P.rows + crow) * row_elems + (int64_t)vi * VPR_ELEMS;
            st16(static_cast<T*>(P.cache_k) + off, z);
            st16(static_cast<T*>(P.cache_v) + off, z);
        }
        return;
    }
    const int rb = (int)blockIdx.x - n_pad;
    const int bl = rb / P.sq;
    const int t = rb - bl * P.sq;
    const ReqParam& rq = P.req[bl];
    const int64_t position = (int64_t)rq.l_req + rq.t0 + t;      // suffix index t0 + t
    const int64_t crow = (int64_t)rq.row_base + rq.n_slots + rq.t0 + t;
    if (threadIdx.x == 0 && l == 0 && crow >= 0 && crow < P.rows) P.pos[crow] = (int32_t)position;
    const int64_t grow = ((int64_t)l * P.batch_total + P.b0 + bl) * P.sq + t;  // tensor row
    const int nq = P.hq * VPH;
    const int items = (P.hq + P.hkv) * VPH;
    const bool row_ok = crow >= 0 && crow < P.rows;
    // item p: query head p / VPH (p < nq) or key/value head (p - nq) / VPH, vector p % VPH
    struct Item {
        uint4 a, b, va, vb;   // the two halves of Q or K, and of V
    };
    auto load = [&](int p, Item& it) {
        const bool is_q = p < nq;
        const int pp = is_q ? p : p - nq;
        const int h = pp / VPH;
        const int iv = pp - h * VPH;
        if (is_q) {
            const T* src = static_cast<const T*>(P.q) + (grow * P.hq + h) * D + iv * E;
            it.a = ld16(src);
            it.b = ld16(src + HALF);
        } else if (row_ok) {
            const int64_t off = (grow * P.hkv + h) * D + iv * E;
            const T* ks = static_cast<const T*>(P.k) + off;
            const T* vs = static_cast<const T*>(P.v) + off;
            it.a = ld16(ks);
            it.b = ld16(ks + HALF);
            it.va = ld16(vs);
            it.vb = ld16(vs + HALF);
        }
    };
    auto store = [&](int p, const Item& it) {
        const bool is_q = p < nq;
        const int pp = is_q ? p : p - nq;
        const int h = pp / VPH;
        const int iv = pp - h * VPH;
        if (!is_q && !row_ok) return;
        float x[E], y[E], gx[E], gy[E];
        V::unpack(it.a, x);
        V::unpack(it.b, y);
        rotate<E>(x, y, cs + iv * E, gx, gy);
        if (is_q) {
            T* dst = static_cast<T*>(P.q_rot) + (grow * P.hq + h) * D + iv * E;
            st16(dst, V::pack(gx));
            st16(dst + HALF, V::pack(gy));
        } else {
            const int64_t coff = ((int64_t)(P.layer0 + l) * P.rows + crow) * row_elems + h * D + iv * E;
            T* kd = static_cast<T*>(P.cache_k) + coff;
            T* vd = static_cast<T*>(P.cache_v) + coff;
            st16(kd, V::pack(gx));
            st16(kd + HALF, V::pack(gy));
            st16(vd, it.va);
            st16(vd + HALF, it.vb);
        }
    };
    // two items per thread per pass, loaded before anything waits on them; the first pass
    // forms the angles in shared memory while its loads are in flight
    const int stride = (int)blockDim.x;
    for (int p0 = 0; p0 < items; p0 += 2 * stride) {
        const int p1 = p0 + (int)threadIdx.x, p2 = p1 + stride;
        Item i1{}, i2{};
        if (p1 < items) load(p1, i1);
        if (p2 < items) load(p2, i2);
        if (p0 == 0) {
            if ((int)threadIdx.x < HALF) cs[threadIdx.x] = turn_cs(P.rope.turn[threadIdx.x], position);
            __syncthreads();
        }
        if (p1 < items) store(p1, i1);
        if (p2 < items) store(p2, i2);
    }
}

int sm_count() {
    int dev = 0, sms = 148;
    if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    return sms;
}

int grid_for(int64_t items, int threads) {
    const int64_t want = (items + threads - 1) / threads;
    const int64_t cap = (int64_t)sm_count() * 8;   // grid-stride beyond 8 CTAs per SM
    return (int)(want < 1 ? 1 : (want > cap ? cap : want));
}

int vph_of(int dtype, int d) { return d / 2 / (dtype == kDtypeBf16 ? 8 : 4); }

}  // namespace

// KERNEL<element type, vectors per half head> for the supported (dtype, head_dim).
#define C2KV_DISPATCH(KERNEL, GRID, PARAMS, DTYPE, D, STREAM)                                  \
    do {                                                                                       \
        if ((DTYPE) == kDtypeBf16 && (D) == 128) KERNEL<__nv_bfloat16, 8><<<GRID, 256, 0, STREAM>>>(PARAMS); \
        else if ((DTYPE) == kDtypeBf16 && (D) == 64) KERNEL<__nv_bfloat16, 4><<<GRID, 256, 0, STREAM>>>(PARAMS); \
        else if ((DTYPE) == kDtypeF32 && (D) == 128) KERNEL<float, 16><<<GRID, 256, 0, STREAM>>>(PARAMS); \
        else if ((DTYPE) == kDtypeF32 && (D) == 64) KERNEL<float, 8><<<GRID, 256, 0, STREAM>>>(PARAMS); \
        else return cudaErrorInvalidValue;                                                     \
    } while (0)

cudaError_t preload_suffix_kernels(int dtype, int d) {
    cudaFuncAttributes fa{};
    if (dtype == kDtypeBf16 && d == 128) return cudaFuncGetAttributes(&fa, suffix_kernel<__nv_bfloat16, 8>);
    if (dtype == kDtypeBf16 && d == 64) return cudaFuncGetAttributes(&fa, suffix_kernel<__nv_bfloat16, 4>);
    if (dtype == kDtypeF32 && d == 128) return cudaFuncGetAttributes(&fa, suffix_kernel<float, 16>);
    if (dtype == kDtypeF32 && d == 64) return cudaFuncGetAttributes(&fa, suffix_kernel<float, 8>);
    return cudaErrorInvalidValue;
}

cudaError_t launch_compose(const ComposeParams& p, int dtype, int d, int layers, cudaStream_t s,
                           int max_ctas) {
    if (p.n_tiles == 0 || p.n_occ == 0) return cudaSuccess;
    (void)cudaGetLastError();   // report this launch's error only, not a stale one
    if (layers > 65535 || p.tile_slots < 1 || p.tile_slots > kComposeTile) return cudaErrorInvalidValue;
    const dim3 grid(max_ctas > 0 && max_ctas < p.n_tiles ? max_ctas : p.n_tiles, layers);
    // one thread per four items of a tile (item = slot, head, vector pair), in whole warps
    const int items = p.tile_slots * p.hkv * vph_of(dtype, d);
    const int threads = std::min(256, std::max(32, (items / 4 + 31) / 32 * 32));
    if (dtype == kDtypeBf16 && d == 128) compose_kernel<__nv_bfloat16, 8><<<grid, threads, 0, s>>>(p);
    else if (dtype == kDtypeBf16 && d == 64) compose_kernel<__nv_bfloat16, 4><<<grid, threads, 0, s>>>(p);
    else if (dtype == kDtypeF32 && d == 128) compose_kernel<float, 16><<<grid, threads, 0, s>>>(p);
    else if (dtype == kDtypeF32 && d == 64) compose_kernel<float, 8><<<grid, threads, 0, s>>>(p);
    else return cudaErrorInvalidValue;
    return cudaGetLastError();
}

cudaError_t launch_compress(const CompressParams& p, int dtype, int d, cudaStream_t s) {
    if (p.m == 0) return cudaSuccess;
    (void)cudaGetLastError();
    const int64_t items = (int64_t)p.m * p.layers * p.hkv * vph_of(dtype, d);
    const int g = grid_for(items, 256);
    C2KV_DISPATCH(compress_kernel, g, p, dtype, d, s);
    return cudaGetLastError();
}

cudaError_t launch_suffix_prep(const SuffixParams& p, int dtype, int d, cudaStream_t s) {
    (void)cudaGetLastError();   // report this launch's error only, not a stale one
    if (p.batch < 1 || p.sq < 1 || p.lq < 1) return cudaSuccess;
    const int64_t blocks = (int64_t)p.batch * p.sq + (p.pad_rows ? (int64_t)p.batch * kPadParts : 0);
    if (blocks > 0x7fffffffLL || p.lq > 65535) return cudaErrorInvalidValue;
    const dim3 grid((unsigned)blocks, p.lq);
    C2KV_DISPATCH(suffix_kernel, grid, p, dtype, d, s);
    return cudaGetLastError();
}

}  // namespace c2kv
