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
#include <atomic>

#include "internal.cuh"
#include "ptx.cuh"
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
template <int N>
struct BulkParams;

// N: the capacity of the launch's occurrence table (a parameter block sized to the launch: a
// launch's latency grows with its parameter bytes).
template <typename T, int VPH, int N>
__global__ void __launch_bounds__(256) compose_kernel(const __grid_constant__ BulkParams<N> P) {
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
// compose, bulk-copy form (every chunk of the launch in the device pool).  A tile is up to
// P.tile_slots consecutive slots of one occurrence in one layer: its K rows and its V rows
// are each one contiguous run of bytes in the pool and one in the cache, so each moves as
// one bulk copy (cp.async.bulk) into shared memory and one back out.  The tiles of all
// layers form one list, layer-major; CTA c (one per SM) takes a contiguous run of it.
//
// Warp 0 is the copy warp: its lane 0 fills every stage of the ring, then per tile waits for
// the turning warps to finish it, stores its K and V, and refills the stage the tile before
// it used (that store's reads of shared memory complete first: wait_group.read 1).  The
// other eight warps turn K in shared memory per tile (thread t always takes the same vector
// of the half-head, so under LOCAL_ROPE storage it forms its E (cos, sin) pairs once per
// occurrence) and write the positions; V passes through untouched.  The occurrence table
// sits in the kernel parameters, sized to the launch (N entries), so a launch of few
// occurrences does not pay for moving a large parameter block.
// ---------------------------------------------------------------------------------------
constexpr int kBulkTurnWarps = 8;
constexpr int kBulkThreads = 32 * (1 + kBulkTurnWarps);
constexpr int kBulkMaxStages = 8;
constexpr uint32_t kBulkSmem = 192u * 1024u;

template <int N>
struct BulkParams : ComposeHead {
    OccParam occ[N];
};

struct BulkTile {
    int32_t layer, src, dst, ns, delta, n, k, j0, ok;
};

__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
                 "l"(src), "r"(bytes), "r"(bar)
                 : "memory");
}
__device__ __forceinline__ void bulk_store(void* dst, uint32_t src, uint32_t bytes) {
    asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(dst), "r"(src), "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ uint4 lds128(uint32_t a) {
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(a));
    return v;
}
__device__ __forceinline__ void sts128(uint32_t a, const uint4& v) {
    asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(a), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
                 : "memory");
}

// A wait that ignores the abort flag (for loads still in flight when the CTA gives up).
__device__ __forceinline__ void mbar_wait_limit(uint32_t bar, uint32_t parity) {
    const long long t0 = clock64();
    while (!mbar_try(bar, parity) && clock64() - t0 < kWaitCycles) {
    }
}

template <typename T, int VPH, int N>
__global__ void __launch_bounds__(kBulkThreads, 1)
    compose_bulk_kernel(const __grid_constant__ BulkParams<N> P, int n_layers, int nst) {
    using V = Vec16<T>;
    constexpr int E = V::N;
    constexpr int HALF = VPH * E;
    constexpr int D = 2 * HALF;
    constexpr int NT = 32 * kBulkTurnWarps;
    static_assert(NT % VPH == 0, "a thread keeps one vector of the half-head");
    extern __shared__ __align__(1024) unsigned char bulk_smem[];
    __shared__ __align__(8) uint64_t full[kBulkMaxStages];
    __shared__ __align__(8) uint64_t turned[kBulkMaxStages];
    __shared__ BulkTile desc[kBulkMaxStages];
    __shared__ uint32_t abort_flag;
    volatile uint32_t* abort = &abort_flag;

    const int tid = (int)threadIdx.x;
    const int ts = P.tile_slots;
    const int64_t row_elems = (int64_t)P.hkv * D;
    const uint32_t row_bytes = (uint32_t)(row_elems * (int64_t)sizeof(T));
    const uint32_t half_stage = (uint32_t)ts * row_bytes;          // K, then V
    const uint32_t sbase = smem_u32(bulk_smem);
    const int64_t total = (int64_t)P.n_tiles * n_layers;
    const int64_t it0 = total * blockIdx.x / gridDim.x;
    const int64_t it1 = total * (blockIdx.x + 1) / gridDim.x;
    const int count = (int)(it1 - it0);
    auto full_bar = [&](int st) { return smem_u32(&full[st]); };
    auto turned_bar = [&](int st) { return smem_u32(&turned[st]); };

    if (tid == 0) {
        abort_flag = 0u;
        for (int st = 0; st < nst; ++st) {
            mbar_init(full_bar(st), 1);
            mbar_init(turned_bar(st), kBulkTurnWarps);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();

    if (tid < 32) {
        // ------------------------------------------------------------- copy warp
        if (tid != 0) return;
        int occ_i = 0, walk_layer = -1;
        auto issue = [&](int i) {
            const int64_t it = it0 + i;
            const int l = (int)(it / P.n_tiles);
            const int tile = (int)(it - (int64_t)l * P.n_tiles);
            if (l != walk_layer) {                // a new layer: find the tile's occurrence
                int lo = 0, hi = P.n_occ - 1;
                while (lo < hi) {
                    const int mid = (lo + hi + 1) >> 1;
                    if (P.occ[mid].tile_base <= tile) lo = mid;
                    else hi = mid - 1;
                }
                occ_i = lo;
                walk_layer = l;
            }
            while (occ_i + 1 < P.n_occ && P.occ[occ_i + 1].tile_base <= tile) ++occ_i;
            const OccParam& o = P.occ[occ_i];
            BulkTile t;
            t.layer = P.layer0 + l;
            t.j0 = (tile - o.tile_base) * ts;
            t.ns = min(ts, o.m - t.j0);
            t.src = o.src_base + t.j0;
            t.dst = o.dest_row + t.j0;
            t.delta = o.delta;
            t.n = o.n;
            t.k = o.k;
            t.ok = t.ns > 0 && t.src >= 0 && (int64_t)t.src + t.ns <= P.pool_slots && t.dst >= 0 &&
                   (int64_t)t.dst + t.ns <= P.rows;
            if (!t.ok && t.ns > 0) atomicOr(P.err, 1);
            const int st = i % nst;
            desc[st] = t;
            const uint32_t bytes = t.ok ? (uint32_t)t.ns * row_bytes : 0u;
            mbar_expect_tx(full_bar(st), 2u * bytes);
            if (t.ok) {
                const int64_t so = ((int64_t)t.layer * P.pool_slots + t.src) * row_elems;
                const uint32_t dk = sbase + (uint32_t)st * 2u * half_stage;
                bulk_load(dk, static_cast<const T*>(P.pool_k) + so, bytes, full_bar(st));
                bulk_load(dk + half_stage, static_cast<const T*>(P.pool_v) + so, bytes, full_bar(st));
            }
        };
        int issued = 0;
        for (; issued < nst && issued < count; ++issued) issue(issued);
        int stored = 0;
        for (; stored < count; ++stored) {
            const int st = stored % nst;
            mbar_wait(turned_bar(st), (uint32_t)(stored / nst) & 1u, P.err, abort);
            if (*abort) break;
            const BulkTile t = desc[st];
            if (t.ok) {
                const int64_t co = ((int64_t)t.layer * P.rows + t.dst) * row_elems;
                const uint32_t bytes = (uint32_t)t.ns * row_bytes;
                const uint32_t dk = sbase + (uint32_t)st * 2u * half_stage;
                bulk_store(static_cast<T*>(P.out_k) + co, dk, bytes);
                bulk_store(static_cast<T*>(P.out_v) + co, dk + half_stage, bytes);
            }
            asm volatile("cp.async.bulk.commit_group;" ::: "memory");
            // the stage of tile `stored - 1` is refilled once that tile's store has read it
            if (stored >= 1 && issued < count) {
                asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory");
                issue(issued++);
            }
        }
        // after an abort: loads in flight land before the CTA leaves; then every store has
        // read shared memory (their writes complete with the grid)
        for (int i = stored; i < issued; ++i) mbar_wait_limit(full_bar(i % nst), (uint32_t)(i / nst) & 1u);
        asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
        return;
    }

    // ----------------------------------------------------------------- turning warps
    const int ct = tid - 32;
    const int lane = tid & 31;
    const int iv = ct % VPH;                  // this thread's vector of the half-head
    float2 cs[E];
    int cs_delta = 0;
    bool cs_valid = false;
    const int per_slot = P.hkv * VPH;
    auto turn_item = [](const float2 (&c)[E], uint4& xv, uint4& yv) {
        float fx[E], fy[E], gx[E], gy[E];
        V::unpack(xv, fx);
        V::unpack(yv, fy);
        rotate<E>(fx, fy, c, gx, gy);
        xv = V::pack(gx);
        yv = V::pack(gy);
    };
    for (int i = 0; i < count; ++i) {
        const int st = i % nst;
        mbar_wait(full_bar(st), (uint32_t)(i / nst) & 1u, P.err, abort);
        if (*abort) break;                    // the same tile for every turning thread
        const BulkTile t = desc[st];
        if (t.ok) {
            const uint32_t dk = sbase + (uint32_t)st * 2u * half_stage;
            if (!P.pre_rope && (!cs_valid || cs_delta != t.delta)) {
#pragma unroll
                for (int e = 0; e < E; ++e) cs[e] = turn_cs(P.rope.turn[iv * E + e], t.delta);
                cs_delta = t.delta;
                cs_valid = true;
            }
            const int items = t.ns * per_slot;
            auto addr = [&](int it) {
                const int sl = it / per_slot;
                const int h = (it - sl * per_slot) / VPH;
                return dk + (uint32_t)sl * row_bytes + (uint32_t)((h * D + iv * E) * (int)sizeof(T));
            };
            auto pre_cs = [&](int it, float2 (&c)[E]) {     // slot j at its composed position delta + p_j
                const int j = t.j0 + it / per_slot;
                const int64_t pos = (int64_t)t.delta + min((j + 1) * t.k, t.n) - 1;
#pragma unroll
                for (int e = 0; e < E; ++e) c[e] = turn_cs(P.rope.turn[iv * E + e], pos);
            };
            constexpr uint32_t YO = HALF * (uint32_t)sizeof(T);
            // two items per pass, both loaded before either is turned
            for (int a0 = ct; a0 < items; a0 += 2 * NT) {
                const int a1 = a0 + NT;
                const bool v1 = a1 < items;
                const uint32_t p0 = addr(a0), p1 = v1 ? addr(a1) : p0;
                uint4 x0 = lds128(p0), y0 = lds128(p0 + YO), x1, y1;
                if (v1) {
                    x1 = lds128(p1);
                    y1 = lds128(p1 + YO);
                }
                if (P.pre_rope) {
                    float2 c0[E];
                    pre_cs(a0, c0);
                    turn_item(c0, x0, y0);
                    if (v1) {
                        float2 c1[E];
                        pre_cs(a1, c1);
                        turn_item(c1, x1, y1);
                    }
                } else {
                    turn_item(cs, x0, y0);
                    if (v1) turn_item(cs, x1, y1);
                }
                sts128(p0, x0);
                sts128(p0 + YO, y0);
                if (v1) {
                    sts128(p1, x1);
                    sts128(p1 + YO, y1);
                }
            }
            if (t.layer == 0)
                for (int sl = ct; sl < t.ns; sl += NT) P.pos[t.dst + sl] = t.delta + min((t.j0 + sl + 1) * t.k, t.n) - 1;
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");   // turned K visible to the copy engine
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(turned_bar(st));
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

template <typename T, int VPH, int N>
cudaError_t launch_bulk_n(const ComposeParams& p, int layers, cudaStream_t s, Hook pre) {
    static std::atomic<uint64_t> attr_set{0};     // per instantiation: devices 0..63 done
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const uint64_t bit = dev < 64 ? (uint64_t)1 << dev : 0;
    if (!(attr_set.load() & bit)) {
        e = cudaFuncSetAttribute(compose_bulk_kernel<T, VPH, N>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)kBulkSmem);
        if (e != cudaSuccess) return e;
        attr_set.fetch_or(bit);
    }
    BulkParams<N> bp;
    static_cast<ComposeHead&>(bp) = p;
    for (int i = 0; i < p.n_occ; ++i) bp.occ[i] = p.occ[i];
    const int64_t row_bytes = (int64_t)p.hkv * VPH * Vec16<T>::N * 2 * (int64_t)sizeof(T);
    const int64_t stage = 2 * (int64_t)p.tile_slots * row_bytes;
    const int nst = (int)std::min<int64_t>(kBulkMaxStages, kBulkSmem / stage);
    if (nst < 2) return cudaErrorInvalidValue;
    const int64_t items = (int64_t)p.n_tiles * layers;
    const int grid = (int)std::min<int64_t>(items, sm_count());
    pre();
    compose_bulk_kernel<T, VPH, N><<<grid, kBulkThreads, (size_t)(nst * stage), s>>>(bp, layers, nst);
    return cudaGetLastError();
}

template <typename T, int VPH>
cudaError_t launch_bulk(const ComposeParams& p, int layers, cudaStream_t s, Hook pre) {
    if (p.n_occ <= 16) return launch_bulk_n<T, VPH, 16>(p, layers, s, pre);
    if (p.n_occ <= 128) return launch_bulk_n<T, VPH, 128>(p, layers, s, pre);
    static_assert(kMaxOcc == 512, "the largest table size is the launch limit");
    return launch_bulk_n<T, VPH, 512>(p, layers, s, pre);
}

// The 16-byte compose kernel with its occurrence table sized to the launch.
template <typename T, int VPH, int N>
cudaError_t launch_16b_n(const ComposeParams& p, dim3 grid, int threads, cudaStream_t s, Hook pre) {
    BulkParams<N> bp;
    static_cast<ComposeHead&>(bp) = p;
    for (int i = 0; i < p.n_occ; ++i) bp.occ[i] = p.occ[i];
    pre();
    compose_kernel<T, VPH, N><<<grid, threads, 0, s>>>(bp);
    return cudaGetLastError();
}

template <typename T, int VPH>
cudaError_t launch_16b(const ComposeParams& p, dim3 grid, int threads, cudaStream_t s, Hook pre) {
    if (p.n_occ <= 16) return launch_16b_n<T, VPH, 16>(p, grid, threads, s, pre);
    if (p.n_occ <= 128) return launch_16b_n<T, VPH, 128>(p, grid, threads, s, pre);
    return launch_16b_n<T, VPH, kMaxOcc>(p, grid, threads, s, pre);
}

cudaError_t launch_compose(const ComposeParams& p, int dtype, int d, int layers, cudaStream_t s,
                           int max_ctas, Hook pre) {
    if (p.n_tiles == 0 || p.n_occ == 0) return cudaSuccess;
    (void)cudaGetLastError();   // report this launch's error only, not a stale one
    if (p.bulk) {
        if (layers < 1 || p.tile_slots < 1 || p.tile_slots > kComposeBulkTile) return cudaErrorInvalidValue;
        for (int i = 0; i < p.n_occ; ++i)
            if (p.occ[i].host) return cudaErrorInvalidValue;
        if (dtype == kDtypeBf16 && d == 128) return launch_bulk<__nv_bfloat16, 8>(p, layers, s, pre);
        if (dtype == kDtypeBf16 && d == 64) return launch_bulk<__nv_bfloat16, 4>(p, layers, s, pre);
        if (dtype == kDtypeF32 && d == 128) return launch_bulk<float, 16>(p, layers, s, pre);
        if (dtype == kDtypeF32 && d == 64) return launch_bulk<float, 8>(p, layers, s, pre);
        return cudaErrorInvalidValue;
    }
    if (layers > 65535 || p.tile_slots < 1 || p.tile_slots > kComposeTile) return cudaErrorInvalidValue;
    const dim3 grid(max_ctas > 0 && max_ctas < p.n_tiles ? max_ctas : p.n_tiles, layers);
    // one thread per four items of a tile (item = slot, head, vector pair), in whole warps
    const int items = p.tile_slots * p.hkv * vph_of(dtype, d);
    const int threads = std::min(256, std::max(32, (items / 4 + 31) / 32 * 32));
    if (dtype == kDtypeBf16 && d == 128) return launch_16b<__nv_bfloat16, 8>(p, grid, threads, s, pre);
    if (dtype == kDtypeBf16 && d == 64) return launch_16b<__nv_bfloat16, 4>(p, grid, threads, s, pre);
    if (dtype == kDtypeF32 && d == 128) return launch_16b<float, 16>(p, grid, threads, s, pre);
    if (dtype == kDtypeF32 && d == 64) return launch_16b<float, 8>(p, grid, threads, s, pre);
    return cudaErrorInvalidValue;
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
