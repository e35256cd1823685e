// Tensor-core attention over [composed cache; suffix] for sm_103a: tcgen05.mma with TMEM
// accumulators, operands staged by TMA in 128-byte-swizzled shared memory.
//
// Work unit (one CTA): two query tiles A and B of 128 packed rows each, consecutive in the
// suffix, of one (layer, request, KV head).  Row m = t * G + g of a tile is suffix token
// t0 + t, query head h_kv * G + g (G = Hq / Hkv), so the G query heads that share a KV
// head form the M dimension of one MMA.  Every K/V tile brought into shared memory feeds
// both tiles' MMAs: 128 KB of MMA work per 64 KB of K/V, which keeps the TMA ingress of an
// SM (about 63 B per clock from L2) below what the tensor core consumes.  The CTA walks
// the request's key tiles of 128 rows (composed slots first, then its own suffix rows);
// only the tiles past S_r + t0 need the causal mask.
//
// Tensor memory (512 columns): S_A [0,128), S_B [128,256), O_A [256,384), O_B [384,512).
// P_x (bf16, two keys per 32-bit column) is written over the first 64 columns of S_x once
// the softmax has read S_x into registers.
//
// The MMA issuer runs, per key tile j,   PV_A(j-1), S_A(j), PV_B(j-1), S_B(j):
// S_A(j) overwrites P_A(j-1) only after PV_A(j-1) in issue order (tcgen05.mma from one
// thread execute in order), and while the softmax of tile A works on S_A(j) the tensor
// core runs PV_B(j-1) and S_B(j), so neither softmax sits on the tensor core's critical
// path as long as it takes less than half a period.  A tcgen05.commit tracks every earlier
// MMA of the thread, so when S_x(j) is reported complete, O_x holds every P.V up to j-1
// and the softmax may rescale it.
//
// Warp roles (384 threads):
//   warp 0      TMA producer: Q_A and Q_B once, then K tiles into a 3-stage ring and V
//               tiles into a 2-stage ring, each issued as soon as its own stage is free (a
//               K stage once S_B has read it, a V stage once P_B.V has).
//   warp 1      MMA issuer (one lane) and TMEM owner.  Warps 2 and 3 only complete
//               warpgroup 0, which hands most of its registers to the softmax warpgroups.
//   warps 4..7  softmax / correction / epilogue of tile A: thread i owns TMEM lane (row) i.
//   warps 8..11 the same for tile B.
//   A softmax thread reads S_j, masks, keeps the running max and sum, rescales O in TMEM
//   only when its row max grew by more than 2^8 (otherwise the stale reference max is
//   kept: the normaliser uses the same one, so the result is exact), and writes P_j.
//
// Every mbarrier wait is bounded (kWaitCycles); on expiry the waiting thread sets bit 1
// of the error word and carries on, so the kernel always terminates and the host reports
// C2KV_ERR_DEVICE_BOUNDS at the next c2kv_sync.
//
// Fused compose + suffix preparation + attention (the same kernel, kFused = true, 512
// threads, the whole step in one launch).  The key tiles come straight from their sources
// instead of the composed cache: the composed slots from the chunk pool, the suffix rows from
// the caller's k_suf / v_suf.  The TMA producer moves whole tiles of one source, and runs of
// 8-row groups of one contiguous source in mixed tiles; the rows of groups that straddle a
// boundary, and the suffix rows of K, are copied by 16-byte cp.async into the same swizzled
// layout, and rows past the suffix are zeroed.  A fourth warpgroup (warps 12..15, the K loaders) turns each composed
// slot's K in shared memory by its occurrence's offset and each suffix row's K by its
// token's position (the compose and suffix kernels' angles and rounding), warp 3 releases
// the V tiles, and the softmax warps, idle until the first S tile, turn the Q tiles in
// shared memory.  In the CTAs of the last query-tile pair (the one whose causal range covers
// the whole suffix) the turned K' and V go to the cache by TMA stores (warp 2 and warp 3)
// with the rows' positions, so the cache is complete for later decode steps.  The pool is
// read once per (layer, request, KV head) and the composed cache written once, rather than
// written by compose and read back by attention.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <math_constants.h>

#include <algorithm>
#include <cstdlib>
#include <cstring>

#include "internal.cuh"
#include "ptx.cuh"
#include "rope.cuh"
#include "vec16.cuh"

namespace c2kv {
namespace {

constexpr int BM = 128;                 // query rows per tile (MMA M)
constexpr int BN = 128;                 // keys per tile (MMA N of S, K of P.V)
constexpr int HD = 128;                 // head dim
constexpr int KSTAGES = 3;              // K ring depth
constexpr int VSTAGES = 2;              // V ring depth
constexpr int TILE = BN * HD * 2;       // bytes of one 128 x 128 bf16 tile (32 KB)
constexpr int HALF_TILE = TILE / 2;     // one 128-byte-wide swizzle column block
constexpr int kThreads = 384;
// Register split (setmaxnreg): warpgroup 0 (TMA producer, MMA issuer, two idle warps) gives
// registers to the two softmax warpgroups.  The kernel is launched with kLaunchRegs per
// thread (the cap that 384 threads leave, 3 warps per SM sub-partition); the split below
// hands out exactly that total, which the host checks against the compiled count.
constexpr int kLaunchRegs = 168;
constexpr int kRegsLow = 136;
constexpr int kRegsHigh = 184;
static_assert(128 * kRegsLow + 256 * kRegsHigh <= kThreads * kLaunchRegs, "register split");
// Fused: 512 threads launch with 128 registers each; the producer/issuer warpgroup and the
// K-loader warpgroup keep 96 each, the softmax warpgroups rise to 160.  (88 / 88 / 168 spilled
// in the first two and measured 7 % slower on the 32-layer step; 88 / 104 / 160 and
// 104 / 104 / 152 fell between.)
constexpr int kThreadsFused = 512;
constexpr int kLaunchRegsFused = 128;
constexpr int kRegsLowFused = 96;       // warps 0..3
constexpr int kRegsLoadFused = 96;      // warps 12..15
constexpr int kRegsHighFused = 160;     // warps 4..11
constexpr int kLoaders = 128;       // K loaders (warps 12..15)
constexpr int kVLoaders = 32;       // V loader (warp 3)
static_assert(128 * kRegsLowFused + 128 * kRegsLoadFused + 256 * kRegsHighFused <=
                  kThreadsFused * kLaunchRegsFused,
              "fused register split");
constexpr uint32_t kTmemCols = 512;     // S_A, S_B, O_A, O_B; P_x over the first half of S_x
constexpr uint32_t kColS = 0, kColO = 256;

// barrier slots
constexpr int B_Q = 0;                   // both Q tiles landed
constexpr int B_KF = 1;                  // + stage
constexpr int B_KE = B_KF + KSTAGES;     // + stage: K stage free (S_A and S_B finished)
constexpr int B_VF = B_KE + KSTAGES;     // + stage
constexpr int B_VE = B_VF + VSTAGES;     // + stage: V stage free (both P.V finished)
constexpr int B_SF = B_VE + VSTAGES;     // + tile: S_x(j) complete (and every MMA before it)
constexpr int B_PF = B_SF + 2;           // + tile: P_x(j) written (and O_x corrected)
constexpr int B_OD = B_PF + 2;           // every MMA finished: O_A, O_B final
constexpr int B_KL = B_OD + 1;           // + stage (fused): the TMA part of a K tile landed
constexpr int B_VL = B_KL + KSTAGES;     // + stage (fused): the TMA part of a V tile landed
constexpr int B_KW = B_VL + VSTAGES;     // + stage (fused): K' of the stage's tile stored to the cache
constexpr int B_VW = B_KW + KSTAGES;     // + stage (fused): V of the stage's tile stored
constexpr int B_QR = B_VW + VSTAGES;     // (fused) Q turned in shared memory
constexpr int B_SK = B_QR + 1;           // (fused) the suffix rows' K' turned into the cache
constexpr int B_QF = B_SK + 1;           // every MMA of a pair has read its Q tiles
constexpr int B_OE = B_QF + 1;           // a pair's epilogue has read O (pairs run in turn)
constexpr int B_WD = B_OE + 1;           // (fused, pairs in turn) the first pair's cache stores done
constexpr int NBAR = B_WD + 1;

constexpr int kSmemTiles = 2 /*Q_A, Q_B*/ + KSTAGES + VSTAGES;
constexpr size_t kSmemBytes = 1024 /*align*/ + (size_t)TILE * kSmemTiles + 8 * NBAR + 16;
static_assert(kSmemBytes <= 232448, "shared memory budget of one sm_100 CTA");

struct TcParams {                // CUtensorMap members carry their own alignment
    CUtensorMap tm_q;        // q_rot   [Lq*Btot][Sq'][Hq][128] box {64, G, TQ, 1}; Sq' = sq_pitch
    CUtensorMap tm_k;        // cache K [L*rows][Hkv][128]      box {64, 1, 128}
    CUtensorMap tm_v;        // cache V, same
    CUtensorMap tm_o;        // out, laid out and boxed like tm_q (the epilogue's TMA stores)
    void* out;
    float* lse;
    int32_t* err;
    int64_t rows;
    int32_t layer0, lq, batch, batch_total, b0, sq, sq_pitch, hq, hkv, group, tq;
    float scale_log2;
    int32_t n_split;
    int32_t pairs;           // pairs of query tiles per (layer, request, KV head)
    int32_t pair_group;      // pairs a CTA runs in turn (1 with key-range splits or fused)
    float* part_o;
    float* part_lse;
    uint32_t* tickets;       // null, or per-unit counters: the last split merges (plain kernel)
    int32_t sif_k;           // 0, or extraction C2 rows with ratio k (plain kernel, one split)
    ReqParam req[kMaxReq];
};

struct FusedTcParams {
    TcParams t;
    // pool [L*pool_slots][Hkv][128] and suffix V [L*Btot*Sq][Hkv][128] in boxes of 128 rows
    // (whole tiles from one source), 64 rows and 8 rows (one swizzle atom) for the runs of
    // clean groups of a mixed tile
    CUtensorMap tm_pk, tm_pv, tm_pk64, tm_pv64, tm_pk8, tm_pv8;
    CUtensorMap tm_sv, tm_sv64, tm_sv8;
    const void* pool_k;      // [L][pool_slots][Hkv][128]
    const void* pool_v;
    const void* k_suf;       // [L][Btot][Sq][Hkv][128], K before RoPE
    const void* v_suf;
    void* cache_k;           // [L][rows][Hkv][128]: written (composed slots, suffix, zero rows)
    void* cache_v;
    int32_t* pos;            // [rows]
    float2* occ_cs;          // scratch [L][occurrences][64]: (cos, sin) of each occurrence's turn
    const float2* sfx_cs;    // [B][Sq][64]: (cos, sin) of each suffix token's position, written
                             // by suffix_angles_kernel (the prerequisite grid)
    int32_t n_occ;           // occurrences of the launch
    int64_t pool_slots;
    RopeTurns rope;
    int32_t req_occ[kMaxFusedReq + 1];
    FusedOcc occ[kMaxFusedOcc];
};

template <bool kFused>
struct KernelParams {
    using type = TcParams;
};
template <>
struct KernelParams<true> {
    using type = FusedTcParams;
};
__device__ __forceinline__ const TcParams& tc_params(const TcParams& p) { return p; }
__device__ __forceinline__ const TcParams& tc_params(const FusedTcParams& p) { return p.t; }

// ------------------------------------------------------------------ tcgen05 wrappers

__device__ __forceinline__ void tc_fence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// Shared-memory matrix descriptor, 128-byte swizzle (layout type 2), sm_100 version bit.
// K-major operands: SBO = 1024 (8 rows of 128 B); LBO unused.  MN-major operands: LBO =
// byte distance between 64-element column blocks, SBO = between 8-row K groups.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
    uint64_t d = 0;
    d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
    d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
    d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
    d |= (uint64_t)1 << 46;
    d |= (uint64_t)2 << 61;
    return d;
}

// Instruction descriptor, kind::f16: D fp32, A and B bf16, A K-major, B K- or MN-major.
__host__ __device__ constexpr uint32_t idesc_bf16(int m, int n, bool b_mn_major) {
    return (1u << 4) | (1u << 7) | (1u << 10) | ((b_mn_major ? 1u : 0u) << 16) |
           ((uint32_t)(n >> 3) << 17) | ((uint32_t)(m >> 4) << 24);
}

__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc,
                                         uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(a), "l"(b), "r"(idesc), "r"(accumulate)
        : "memory");
}

// Same, with A read from tensor memory (rows in lanes, K packed two bf16 per column).
__device__ __forceinline__ void mma_bf16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b,
                                            uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
        "r"(a_tmem), "l"(b), "r"(idesc), "r"(accumulate)
        : "memory");
}

__device__ __forceinline__ void mma_commit(uint32_t bar) {
    asm volatile(
        "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
        : "memory");
}

// 32 consecutive TMEM columns of this thread's lane -> 32 registers.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&v)[32]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
        "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
        : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]),
          "=r"(v[7]), "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]),
          "=r"(v[13]), "=r"(v[14]), "=r"(v[15]), "=r"(v[16]), "=r"(v[17]), "=r"(v[18]),
          "=r"(v[19]), "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]), "=r"(v[24]),
          "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]),
          "=r"(v[31])
        : "r"(taddr));
}

__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&v)[16]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];"
        : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]),
          "=r"(v[7]), "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]),
          "=r"(v[13]), "=r"(v[14]), "=r"(v[15])
        : "r"(taddr));
}

__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&v)[16]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
        "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16};" ::"r"(taddr),
        "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]),
        "r"(v[8]), "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]),
        "r"(v[15])
        : "memory");
}

__device__ __forceinline__ void tmem_ld_wait() {
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_st_wait() {
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

// 2^x on the MUFU pipe (ex2.approx: relative error ~2^-22, flushes subnormal results,
// 2^-inf = +0).
__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&v);
}

// Two fp32 lanes per instruction (sm_100 packed f32x2 arithmetic, round to nearest: each
// lane is bitwise the scalar fmaf / add), and the three-input maximum.
__device__ __forceinline__ void ffma2(float& d0, float& d1, float a0, float a1, float b, float c) {
    asm("{\n\t.reg .b64 pa, pb, pc, pd;\n\t"
        "mov.b64 pa, {%2, %3};\n\t"
        "mov.b64 pb, {%4, %4};\n\t"
        "mov.b64 pc, {%5, %5};\n\t"
        "fma.rn.f32x2 pd, pa, pb, pc;\n\t"
        "mov.b64 {%0, %1}, pd;\n\t}"
        : "=f"(d0), "=f"(d1)
        : "f"(a0), "f"(a1), "f"(b), "f"(c));
}

__device__ __forceinline__ void fadd2(float& d0, float& d1, float a0, float a1) {
    asm("{\n\t.reg .b64 pa, pd;\n\t"
        "mov.b64 pa, {%2, %3};\n\t"
        "mov.b64 pd, {%0, %1};\n\t"
        "add.rn.f32x2 pd, pd, pa;\n\t"
        "mov.b64 {%0, %1}, pd;\n\t}"
        : "+f"(d0), "+f"(d1)
        : "f"(a0), "f"(a1));
}

__device__ __forceinline__ float fmax3(float a, float b, float c) {
    float d;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
}

// A 4-D tile of shared memory to global memory by TMA (bulk async-group of the thread).
__device__ __forceinline__ void tma_store_4d(const CUtensorMap* tm, uint32_t src, int c0, int c1, int c2, int c3) {
    asm volatile("cp.async.bulk.tensor.4d.global.shared::cta.bulk_group [%0, {%1, %2, %3, %4}], [%5];" ::"l"(
                     reinterpret_cast<uint64_t>(tm)),
                 "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(src)
                 : "memory");
}
// 32 bytes (one full L2 sector) to global memory in one instruction (sm_100 256-bit stores).
__device__ __forceinline__ void stg256(void* p, const uint32_t* w) {
    asm volatile("st.global.v8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};" ::"l"(p), "r"(w[0]), "r"(w[1]),
                 "r"(w[2]), "r"(w[3]), "r"(w[4]), "r"(w[5]), "r"(w[6]), "r"(w[7])
                 : "memory");
}
__device__ __forceinline__ void sts128_(uint32_t a, const uint4& v) {
    asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(a), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
                 : "memory");
}

// Splits merged inside the kernel (TcParams::tickets).  Every split CTA of a (layer, request,
// KV head, pair) unit writes its normalised fp32 partial and log2-domain lse, then both softmax
// warpgroups meet (named barrier 4); one thread releases the partials (a GPU-scope fence) and
// takes a ticket.  In the CTA that takes the last one, warpgroup A merges every row of the
// pair as attn_combine_kernel does: 32 threads a row, 4 channels each, eight splits' lse and
// output slices loaded before any is used; lse = log2 sum_s 2^lse_s,
// O = sum_s 2^(lse_s - lse) O_s.  Then the counter goes back to zero for the next launch.  No
// thread waits on another CTA.  At most kMaxMergeSplits splits (the host merges by launch
// beyond that).
__device__ __forceinline__ void split_merge(const TcParams& P, uint32_t sBar, int x, int r, int t0, int l,
                                            int b, int hk) {
    __threadfence();
    asm volatile("bar.sync 4, 256;" ::: "memory");
    const uint32_t sFlag = sBar + 8u * (uint32_t)NBAR + 8u;     // spare word after the barriers
    const int n_groups = (int)(gridDim.x / P.n_split);
    const int64_t unit = ((int64_t)blockIdx.z * gridDim.y + blockIdx.y) * n_groups + blockIdx.x / P.n_split;
    if (x == 0 && r == 0) {
        __threadfence();
        const uint32_t t = atomicAdd(P.tickets + unit, 1u);
        asm volatile("st.shared.u32 [%0], %1;" ::"r"(sFlag), "r"(t == (uint32_t)(P.n_split - 1) ? 1u : 0u) : "memory");
    }
    asm volatile("bar.sync 4, 256;" ::: "memory");
    uint32_t last;
    asm volatile("ld.shared.u32 %0, [%1];" : "=r"(last) : "r"(sFlag) : "memory");
    if (!last || x != 0) return;
    __threadfence();                                 // the other splits' partials are visible
    const int G = P.group, tq = P.tq;
    const int t0a = t0, t0b = t0 + tq;               // (warpgroup A's tile is tile A)
    const int rows_a = min(BM, (P.sq - t0a) * G);
    const int rows_b = t0b < P.sq ? min(BM, (P.sq - t0b) * G) : 0;
    const int64_t part_rows = (int64_t)P.lq * P.batch_total * P.sq * P.hq;
    const int ns = P.n_split;
#pragma unroll 1
    for (int it = r; it < (rows_a + rows_b) * 32; it += BM) {
        const int row = it >> 5, c4 = it & 31;
        const int xr = row < rows_a ? 0 : 1, rr = row - xr * rows_a;
        const int t = (xr ? t0b : t0a) + rr / G, g = rr - (rr / G) * G;
        const int64_t row_id = (((int64_t)l * P.batch_total + b) * P.sq_pitch + t) * P.hq + hk * G + g;
        const int64_t lse_id = (((int64_t)l * P.batch_total + b) * P.hq + hk * G + g) * P.sq_pitch + t;
        constexpr int SB = 8;                        // splits in flight together
        float mx = -CUDART_INF_F;
#pragma unroll 1
        for (int s0 = 0; s0 < ns; s0 += SB) {
#pragma unroll
            for (int s = s0; s < s0 + SB; ++s)
                if (s < ns) mx = fmaxf(mx, __ldcg(P.part_lse + (int64_t)s * part_rows + lse_id));
        }
        float wsum = 0.f;
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 1
        for (int s0 = 0; s0 < ns; s0 += SB) {
            float ls[SB];
            float4 o[SB];
#pragma unroll
            for (int i = 0; i < SB; ++i) {
                ls[i] = -CUDART_INF_F;
                o[i] = make_float4(0.f, 0.f, 0.f, 0.f);
                if (s0 + i < ns) {
                    ls[i] = __ldcg(P.part_lse + (int64_t)(s0 + i) * part_rows + lse_id);
                    o[i] = __ldcg(reinterpret_cast<const float4*>(P.part_o + ((int64_t)(s0 + i) * part_rows + row_id) * HD) + c4);
                }
            }
#pragma unroll
            for (int i = 0; i < SB; ++i) {
                const float w = ls[i] == -CUDART_INF_F ? 0.f : ex2(ls[i] - mx);
                acc.x += w * o[i].x;
                acc.y += w * o[i].y;
                acc.z += w * o[i].z;
                acc.w += w * o[i].w;
                wsum += w;
            }
        }
        const float inv = 1.0f / wsum;
        uint2 pk;
        pk.x = pack_bf16(acc.x * inv, acc.y * inv);
        pk.y = pack_bf16(acc.z * inv, acc.w * inv);
        *reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(P.out) + row_id * HD + c4 * 4) = pk;
        if (P.lse != nullptr && c4 == 0) P.lse[lse_id] = (mx + log2f(wsum)) * 0.69314718055994531f;
    }
    if (r == 0) P.tickets[unit] = 0u;
}

// The query tokens and key tiles of pair pr of query tiles (split sp of its key range).  The
// key tiles are, in order: tile 0 if lead0, then n_mid tiles from j_base, then the rest from
// j_tail; a plain pair's are the n_kv tiles from j_base (lead0 = false, n_mid = n_kv).
struct PairSpan {
    int t0a, t0b;       // first suffix token of tile A, of tile B
    bool has_b;
    int t_last;         // last suffix token of the pair
    int j_base, n_kv;   // this split's key tiles: n_kv of them, the first run from j_base
    bool lead0;
    int n_mid, j_tail;
};
// Bit i set for the keys lo + i (i < 32) that lie in [a, b).
__device__ __forceinline__ uint32_t range_bits(int lo, int a, int b) {
    const int x = max(a - lo, 0), y = min(b - lo, 32);
    if (y <= x) return 0u;                                   // (so x < 32 below)
    const uint32_t below_y = y >= 32 ? 0xffffffffu : (1u << y) - 1u;
    return below_y & ~((1u << x) - 1u);
}

// The box of a tensor map at the given coordinates into L2 (no shared memory, no barrier).
__device__ __forceinline__ void tma_prefetch_3d(const CUtensorMap* tm, int c0, int c1, int c2) {
    asm volatile("cp.async.bulk.prefetch.tensor.3d.L2.global.tile [%0, {%1, %2, %3}];"
                 ::"l"(reinterpret_cast<uint64_t>(tm)), "r"(c0), "r"(c1), "r"(c2) : "memory");
}
__device__ __forceinline__ void tma_prefetch_4d(const CUtensorMap* tm, int c0, int c1, int c2, int c3) {
    asm volatile("cp.async.bulk.prefetch.tensor.4d.L2.global.tile [%0, {%1, %2, %3, %4}];"
                 ::"l"(reinterpret_cast<uint64_t>(tm)), "r"(c0), "r"(c1), "r"(c2), "r"(c3) : "memory");
}

// Key tile of the pair's i-th key tile.
__device__ __forceinline__ int span_tile(const PairSpan& o, int i) {
    const int i1 = i - (o.lead0 ? 1 : 0);
    return i1 < 0 ? 0 : i1 < o.n_mid ? o.j_base + i1 : o.j_tail + (i1 - o.n_mid);
}
__device__ __forceinline__ PairSpan pair_span(const TcParams& P, int pr, int sp, int s_r) {
    PairSpan o;
    o.t0a = 2 * pr * P.tq;
    o.t0b = o.t0a + P.tq;
    o.has_b = o.t0b < P.sq;
    o.t_last = min(P.sq - 1, (o.has_b ? o.t0b : o.t0a) + P.tq - 1);
    o.lead0 = false;
    if (P.sif_k > 0) {
        // extraction C2 rows c_j, j in [t0a, t_last], over a chunk of n = s_r document keys:
        // the tiles of their blocks' document keys, tile 0 (the sink block) if not among
        // them, then the tiles of the C2 keys c_0 .. c_{t_last} at rows n .. n + t_last not
        // already taken (every C2 block holds at least one document token, jk < n)
        const int k = P.sif_k, n = s_r;
        const int b0 = (o.t0a * k) / BN, b1 = (min((o.t_last + 1) * k, n) - 1) / BN;
        const int c0 = max(n / BN, b1 + 1), c1 = (n + o.t_last) / BN;
        o.lead0 = b0 > 0;
        o.j_base = b0;
        o.n_mid = b1 - b0 + 1;
        o.j_tail = c0;
        o.n_kv = (o.lead0 ? 1 : 0) + o.n_mid + max(0, c1 - c0 + 1);
        return o;
    }
    const int n_kv_all = (s_r + o.t_last + 1 + BN - 1) / BN;
    const int per_split = (n_kv_all + P.n_split - 1) / P.n_split;
    o.j_base = sp * per_split;
    o.n_kv = max(0, min(n_kv_all, o.j_base + per_split) - o.j_base);
    o.n_mid = o.n_kv;
    o.j_tail = o.j_base + o.n_kv;
    return o;
}

// ------------------------------------------------------------------ kernel

// One softmax thread's work on tile x (A or B) for every key tile of a pair, then its
// epilogue.  r = TMEM lane (row within the tile), t0 = first suffix token of the tile.
// sf_base: S_x tiles completed in earlier pairs (phase count); od_par: the phase of B_OD that
// closes this pair; arrive_oe: tell the issuer (B_OE) once O has been read, when the CTA
// runs further pairs.  stage: the Q tiles' shared memory when this is the CTA's last pair
// (no further Q will land there), else 0: O then leaves through it, the tile's rows written
// in the 128-byte-swizzled layout and stored by TMA, instead of 16-byte stores of a row per
// thread (which touch a separate cache line per thread).
// kMerge: the plain kernel, whose split partials may be merged in the kernel (split_merge).
// kSif: the plain kernel over extraction C2 rows (TcParams::sif_k), its own instantiation.
// kKpp: the plain kernel's decode instantiation, whose pairs with one query tile split their
// key tiles between the two warpgroups (kpp: this pair does).
template <bool kMerge, bool kSif = false, bool kKpp = false>
__device__ __forceinline__ void softmax_tile(const TcParams& P, uint32_t tmem, uint32_t sBar, int x,
                                            int quad, int lane, int t0, int l, int bl, int b,
                                            int hk, int sp, const PairSpan& span, uint32_t sf_base,
                                            uint32_t od_par, bool arrive_oe,
                                            volatile uint32_t* abort, uint32_t stage = 0u,
                                            bool kpp_pair = false) {
    auto bar = [&](int i) { return sBar + 8u * (uint32_t)i; };
    const int G = P.group;
    // keys before the launch's first query token: the composed slots and, for a decode step
    // (t0 > 0), the suffix rows written before it
    const int s_r = P.req[bl].n_slots + P.req[bl].t0;
    const int r = quad * 32 + lane;                 // row = TMEM lane
    const uint32_t lane_addr = (uint32_t)(quad * 32) << 16;
    const uint32_t colS = kColS + (uint32_t)x * BN;  // S_x, and P_x over its first 64 columns
    const uint32_t colO = kColO + (uint32_t)x * HD;
    const int t_row = min(t0 + r / G, P.sq - 1);    // rows past the suffix mirror its end
    const int lim = s_r + t_row;                    // last key this row may see
    const float sc = P.scale_log2;
    const int n_kv = span.n_kv;
    float m_run = -CUDART_INF_F;
    float l_run = 0.f;

    // kpp: this warpgroup takes every other key tile (x, x + 2, ...) of the pair's one query
    // tile; i counts the tiles it has taken
    const bool kpp = kKpp && kpp_pair;
    for (int j = kpp ? x : 0, i = 0; j < n_kv; j += kpp ? 2 : 1, ++i) {
        mbar_wait(bar(B_SF + x), (sf_base + (uint32_t)i) & 1u, P.err, abort);
        tc_fence_after();
        uint32_t sv[4][32];
#pragma unroll
        for (int c = 0; c < 4; ++c) tmem_ld32(tmem + lane_addr + colS + c * 32, sv[c]);
        tmem_ld_wait();

        const int kbase = (kSif ? span_tile(span, j) : span.j_base + j) * BN;
        if (kbase + BN - 1 > lim) {
#pragma unroll
            for (int c = 0; c < 4; ++c)
#pragma unroll
                for (int e = 0; e < 32; ++e)
                    if (kbase + c * 32 + e > lim) sv[c][e] = __float_as_uint(-CUDART_INF_F);
        }
        if constexpr (kSif) {
            // extraction C2 row c_{t_row}: of the document keys (rows below s_r) it sees the
            // sink block [0, min(k, n)) and its own block [t_row k, min((t_row + 1) k, n)); per
            // 32-key chunk, the bits of the keys that stay (those two blocks and the C2 keys)
            if (kbase < s_r) {
                const int sink = min(P.sif_k, s_r);
                const int blo = t_row * P.sif_k, bhi = min(blo + P.sif_k, s_r);
#pragma unroll
                for (int c = 0; c < 4; ++c) {
                    const int lo = kbase + c * 32;
                    const uint32_t keep = range_bits(lo, 0, sink) | range_bits(lo, blo, bhi) |
                                          range_bits(lo, s_r, lo + 32);
#pragma unroll
                    for (int e = 0; e < 32; ++e)
                        if (!(keep & (1u << e))) sv[c][e] = __float_as_uint(-CUDART_INF_F);
                }
            }
        }
        // row max: three-input maxima, one chain per 32-column chunk
        float mx4[4];
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            float m = fmaxf(__uint_as_float(sv[c][0]), __uint_as_float(sv[c][1]));
#pragma unroll
            for (int e = 2; e < 32; e += 2)
                m = fmax3(m, __uint_as_float(sv[c][e]), __uint_as_float(sv[c][e + 1]));
            mx4[c] = m;
        }
        const float mx = fmaxf(fmaxf(mx4[0], mx4[1]), fmaxf(mx4[2], mx4[3]));
        const float m_new = fmaxf(m_run, mx * sc);
        const bool resc = m_new > m_run + 8.0f;       // false while nothing is visible
        const float m_use = resc ? m_new : m_run;
        const float alpha = resc ? ex2(m_run - m_new) : 1.0f;
        const float m_sub = m_use == -CUDART_INF_F ? 0.f : m_use;   // all masked so far

        // S_x(j) complete implies the P_x.V before it complete: O_x is current and may be scaled
        if (i >= 1 && __any_sync(0xffffffffu, resc)) {
#pragma unroll 1
            for (int c = 0; c < 8; ++c) {
                uint32_t ov[16];
                tmem_ld16(tmem + lane_addr + colO + c * 16, ov);
                tmem_ld_wait();
#pragma unroll
                for (int e = 0; e < 16; ++e) ov[e] = __float_as_uint(__uint_as_float(ov[e]) * alpha);
                tmem_st16(tmem + lane_addr + colO + c * 16, ov);
            }
        }
        float ps[4];                                   // two packed accumulators
#pragma unroll
        for (int e = 0; e < 4; ++e) ps[e] = 0.f;
        // P_j (bf16, keys 2c and 2c+1 packed in column c) over the first half of S_x
        const uint32_t p_addr = tmem + lane_addr + colS;
        const float neg_m = -m_sub;
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            uint32_t pk[16];
#pragma unroll
            for (int e = 0; e < 32; e += 2) {
                float a0, a1;
                ffma2(a0, a1, __uint_as_float(sv[c][e]), __uint_as_float(sv[c][e + 1]), sc, neg_m);
                a0 = ex2(a0);
                a1 = ex2(a1);
                if (e & 2) fadd2(ps[2], ps[3], a0, a1); else fadd2(ps[0], ps[1], a0, a1);
                pk[e >> 1] = pack_bf16(a0, a1);
            }
            tmem_st16(p_addr + (uint32_t)c * 16u, pk);
        }
        tmem_st_wait();
        const float sum = (ps[0] + ps[1]) + (ps[2] + ps[3]);
        l_run = l_run * alpha + sum;
        m_run = m_use;
        tc_fence_before();
        mbar_arrive(bar(B_PF + x));
    }

    if (kKpp && kpp) {
        // the two halves meet: B leaves its row's (m, l) in the Q_B tile (unused with one
        // query tile), and A, once every MMA is done, folds O_B into O_A in TMEM with the
        // exact rule (log2 domain, each half against its own reference maximum)
        //     m = max(m_A, m_B),  w_x = 2^(m_x - m),  l = w_A l_A + w_B l_B,  O = w_A O_A + w_B O_B
        const uint32_t xch = stage + (uint32_t)TILE + (uint32_t)r * 8u;
        if (x == 1) {
            asm volatile("st.shared.v2.f32 [%0], {%1, %2};" ::"r"(xch), "f"(m_run), "f"(l_run) : "memory");
            asm volatile("bar.sync 4, 256;" ::: "memory");
            if constexpr (kMerge)
                if (P.n_split > 1 && P.tickets != nullptr) split_merge(P, sBar, x, r, t0, l, b, hk);
            if (arrive_oe) {
                tc_fence_before();
                mbar_arrive(bar(B_OE));
            }
            return;
        }
        mbar_wait(bar(B_OD), od_par, P.err, abort);
        tc_fence_after();
        asm volatile("bar.sync 4, 256;" ::: "memory");
        float m_b, l_b;
        asm volatile("ld.shared.v2.f32 {%0, %1}, [%2];" : "=f"(m_b), "=f"(l_b) : "r"(xch) : "memory");
        const float m = fmaxf(m_run, m_b);
        const float w_a = l_run > 0.f ? ex2(m_run - m) : 0.f;
        const float w_b = l_b > 0.f ? ex2(m_b - m) : 0.f;
        const uint32_t colO_b = kColO + HD;
#pragma unroll 1
        for (int c = 0; c < 8; ++c) {
            uint32_t oa[16], ob[16];
            tmem_ld16(tmem + lane_addr + colO + c * 16, oa);
            tmem_ld16(tmem + lane_addr + colO_b + c * 16, ob);
            tmem_ld_wait();
#pragma unroll
            for (int e = 0; e < 16; ++e) {
                const float va = w_a != 0.f ? w_a * __uint_as_float(oa[e]) : 0.f;   // (an empty half's O
                const float vb = w_b != 0.f ? w_b * __uint_as_float(ob[e]) : 0.f;   //  is never read)
                oa[e] = __float_as_uint(va + vb);
            }
            tmem_st16(tmem + lane_addr + colO + c * 16, oa);
        }
        tmem_st_wait();
        l_run = w_a * l_run + w_b * l_b;
        m_run = m;
    }

    // ---------------------------------------------------------------- epilogue
    if (n_kv > 0) {
        mbar_wait(bar(B_OD), od_par, P.err, abort);
        tc_fence_after();
    }
    const int t = t0 + r / G;
    const int g = r - (r / G) * G;
    const bool any = l_run > 0.f;                 // some key of this split was visible
    const float inv = any ? 1.0f / l_run : 0.f;
    const int64_t row_id = (((int64_t)l * P.batch_total + b) * P.sq_pitch + t) * P.hq + hk * G + g;
    const int64_t lse_id = (((int64_t)l * P.batch_total + b) * P.hq + hk * G + g) * P.sq_pitch + t;
    if (P.n_split == 1 && stage != 0u && n_kv > 0) {
        const uint32_t sbase = stage + (uint32_t)x * TILE;
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            uint32_t ov[32];
            tmem_ld32(tmem + lane_addr + colO + c * 32, ov);
            tmem_ld_wait();
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                uint4 w;
                w.x = pack_bf16(__uint_as_float(ov[k * 8 + 0]) * inv, __uint_as_float(ov[k * 8 + 1]) * inv);
                w.y = pack_bf16(__uint_as_float(ov[k * 8 + 2]) * inv, __uint_as_float(ov[k * 8 + 3]) * inv);
                w.z = pack_bf16(__uint_as_float(ov[k * 8 + 4]) * inv, __uint_as_float(ov[k * 8 + 5]) * inv);
                w.w = pack_bf16(__uint_as_float(ov[k * 8 + 6]) * inv, __uint_as_float(ov[k * 8 + 7]) * inv);
                const int q = c * 4 + k;                       // 16-byte chunk of the row
                sts128_(sbase + (uint32_t)((q >> 3) * HALF_TILE + r * 128 + (((q & 7) ^ (r & 7)) << 4)), w);
            }
        }
        if (P.lse != nullptr && t < P.sq)
            P.lse[lse_id] = (m_run + log2f(l_run)) * 0.69314718055994531f;
        if (arrive_oe) {
            tc_fence_before();
            mbar_arrive(bar(B_OE));
        }
        // the rows visible to the TMA engine, every row of the tile written, then one store of
        // both 64-column halves (tokens past the suffix fall outside the map and are dropped)
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        asm volatile("bar.sync %0, 128;" ::"r"(2 + x) : "memory");
        if (r == 0) {
            const int qz = l * P.batch_total + b;
            tma_store_4d(&P.tm_o, sbase, 0, hk * G, t0, qz);
            tma_store_4d(&P.tm_o, sbase + HALF_TILE, 64, hk * G, t0, qz);
            asm volatile("cp.async.bulk.commit_group;" ::: "memory");
            // the CTA may leave once the store has read shared memory; its writes complete
            // with the grid
            asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
        }
        return;
    }
    if (P.n_split == 1) {
        // each thread writes its own row, a full 32-byte sector per store: the lanes of a
        // warp hold rows of up to 32 different lines, so a narrower store would leave every
        // sector it touches half written
        // (rows are 256 bytes apart, so the output's base alignment decides; the entry points
        // guarantee 16 bytes only)
        __nv_bfloat16* orow = static_cast<__nv_bfloat16*>(P.out) + row_id * HD;
        const bool a32 = (reinterpret_cast<uintptr_t>(P.out) & 31u) == 0;
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            uint32_t ov[32];
            tmem_ld32(tmem + lane_addr + colO + c * 32, ov);
            tmem_ld_wait();
            if (t < P.sq) {
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    uint32_t w[8];
#pragma unroll
                    for (int e = 0; e < 8; ++e)
                        w[e] = pack_bf16(__uint_as_float(ov[h * 16 + 2 * e]) * inv,
                                         __uint_as_float(ov[h * 16 + 2 * e + 1]) * inv);
                    if (a32) {
                        stg256(orow + c * 32 + h * 16, w);
                    } else {
                        *reinterpret_cast<uint4*>(orow + c * 32 + h * 16) = make_uint4(w[0], w[1], w[2], w[3]);
                        *reinterpret_cast<uint4*>(orow + c * 32 + h * 16 + 8) = make_uint4(w[4], w[5], w[6], w[7]);
                    }
                }
            }
        }
        if (P.lse != nullptr && t < P.sq)
            P.lse[lse_id] = (m_run + log2f(l_run)) * 0.69314718055994531f;
    } else {
        // partial over this split's keys: normalised O (fp32) and its log2-domain lse
        const int64_t part_rows = (int64_t)P.lq * P.batch_total * P.sq * P.hq;
        float* orow = P.part_o + ((int64_t)sp * part_rows + row_id) * HD;
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            uint32_t ov[32];
            if (n_kv > 0) {
                tmem_ld32(tmem + lane_addr + colO + c * 32, ov);
                tmem_ld_wait();
            } else {
#pragma unroll
                for (int e = 0; e < 32; ++e) ov[e] = 0u;
            }
            if (t < P.sq) {
#pragma unroll
                for (int q8 = 0; q8 < 4; ++q8) {
                    uint32_t w[8];
#pragma unroll
                    for (int e = 0; e < 8; ++e) w[e] = __float_as_uint(__uint_as_float(ov[q8 * 8 + e]) * inv);
                    stg256(orow + c * 32 + q8 * 8, w);
                }
            }
        }
        if (t < P.sq)
            P.part_lse[(int64_t)sp * part_rows + lse_id] = any ? m_run + log2f(l_run) : -CUDART_INF_F;
        if constexpr (kMerge)
            if (P.tickets != nullptr) split_merge(P, sBar, x, r, t0, l, b, hk);
    }
    if (arrive_oe) {          // O has been read out of TMEM: the next pair may overwrite it
        tc_fence_before();
        mbar_arrive(bar(B_OE));
    }
}

// The MMA issuer (one thread).  The tensor core's queue holds about one MMA, so anything
// the issuing thread does between two MMAs idles it, and a branch there costs about as much
// as an MMA.  So the descriptors are precomputed, the issue blocks are straight-line code,
// the kernel is specialised on whether the CTA has a tile B, and the ring stages and
// barrier parities advance by selects rather than branches.  Each block waits for its own
// inputs only: waiting for a later block's P inside an S block would hold that S back until
// the other tile's softmax finished, putting the two softmaxes in series.
// Ring positions and phase counts that carry over from one pair of query tiles to the next
// when a CTA runs several pairs of one (layer, request, KV head) in turn.
struct RingState {
    int ks = 0;               // K stage of the next K tile, and its fill parity
    uint32_t kph = 0u;
    int vs = 0;               // V stage of the next V tile, and its fill parity
    uint32_t vph = 0u;
    uint32_t pa = 0u, pb = 0u;    // P_A, P_B tiles completed in earlier pairs
};

// The MMA issuer for one pair of query tiles (n_kv >= 1 key tiles).  q_ready / q_par: the
// barrier phase that says Q is in shared memory.  wait_oe: a previous pair's epilogue must
// have read O (phase oe_par of B_OE) before this pair's first P.V overwrites it.  B_QF says
// that every S of the pair has read Q, and B_OD at the end that O is final.
template <bool kHasB>
__device__ __forceinline__ void mma_issuer(const TcParams& P, uint32_t tmem, uint32_t sQ, uint32_t sK,
                                           uint32_t sV, uint32_t sBar, int n_kv, int q_ready,
                                           uint32_t q_par, RingState& st, bool wait_oe, uint32_t oe_par,
                                           volatile uint32_t* abort) {
    static_assert(KSTAGES == 3 && VSTAGES == 2, "the issue schedule assumes 3 K and 2 V stages");
    auto bar = [&](int i) { return sBar + 8u * (uint32_t)i; };
    constexpr uint32_t idS = idesc_bf16(BM, BN, false);
    constexpr uint32_t idO = idesc_bf16(BM, HD, true);
    constexpr uint64_t kTileDesc = (uint64_t)(TILE >> 4);     // one tile in descriptor units
    // descriptors of tile bases; a K step adds its byte offset / 16 to the low field
    const uint64_t dQa = sw128_desc(sQ, 16, 1024);
    const uint64_t dQb = sw128_desc(sQ + TILE, 16, 1024);
    const uint64_t dK0 = sw128_desc(sK, 16, 1024);
    const uint64_t dV0 = sw128_desc(sV, HALF_TILE, 1024);
    const uint32_t tS_a = tmem + kColS, tS_b = tmem + kColS + BN;
    const uint32_t tO_a = tmem + kColO, tO_b = tmem + kColO + HD;

    // S = Q K^T (8 K steps of 16)
    auto s_block = [&](uint64_t dq, uint64_t dk, uint32_t d) {
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk) {
            const uint64_t off = (uint64_t)(((kk >> 2) * HALF_TILE + (kk & 3) * 32) >> 4);
            mma_bf16(d, dq + off, dk + off, idS, kk > 0 ? 1u : 0u);
        }
    };
    // O += P V with P (bf16 pairs) from TMEM: 16 keys (8 columns) per step; the first step
    // of the first block overwrites O
    auto pv_block = [&](uint32_t p, uint64_t dv, uint32_t o, uint32_t acc0) {
#pragma unroll
        for (int kk = 0; kk < BN / 16; ++kk)
            mma_bf16_ts(o, p + (uint32_t)kk * 8u, dv + (uint64_t)((kk * 2048) >> 4), idO,
                        kk > 0 ? 1u : acc0);
    };
    auto wait = [&](int i, uint32_t parity) {
        mbar_wait(bar(i), parity, P.err, abort);
        tc_fence_after();
    };
    auto next_k = [&]() {
        const bool w = st.ks == KSTAGES - 1;
        st.ks = w ? 0 : st.ks + 1;
        st.kph ^= w ? 1u : 0u;
    };
    auto next_v = [&]() {
        const bool w = st.vs == VSTAGES - 1;
        st.vs = w ? 0 : st.vs + 1;
        st.vph ^= w ? 1u : 0u;
    };
    // one key tile j >= 1:  PV_A(j-1)  S_A(j)  PV_B(j-1)  S_B(j)
    //   st.ks, st.kph: K stage and fill parity of tile j;  st.vs, st.vph: V stage and parity
    //   of tile j-1;  ppa, ppb: parities of P_A(j-1), P_B(j-1);  acc0: 0 only for the first
    //   P.V of the pair (j == 1), which also waits for the previous epilogue when asked
    auto tile = [&](uint32_t ppa, uint32_t ppb, uint32_t acc0, bool oe) {
        const uint64_t dk = dK0 + (uint64_t)st.ks * kTileDesc;
        const uint64_t dv = dV0 + (uint64_t)st.vs * kTileDesc;
        wait(B_PF + 0, ppa);
        wait(B_VF + st.vs, st.vph);
        if (oe) wait(B_OE, oe_par);
        pv_block(tS_a, dv, tO_a, acc0);
        wait(B_KF + st.ks, st.kph);
        s_block(dQa, dk, tS_a);
        mma_commit(bar(B_SF + 0));
        if (kHasB) {
            wait(B_PF + 1, ppb);
            pv_block(tS_b, dv, tO_b, acc0);
        }
        mma_commit(bar(B_VE + st.vs));
        if (kHasB) {
            s_block(dQb, dk, tS_b);
            mma_commit(bar(B_SF + 1));
        }
        mma_commit(bar(B_KE + st.ks));
    };

    wait(q_ready, q_par);
    wait(B_KF + st.ks, st.kph);
    // key tile 0: S_A(0), S_B(0)
    const uint64_t dk0 = dK0 + (uint64_t)st.ks * kTileDesc;
    s_block(dQa, dk0, tS_a);
    mma_commit(bar(B_SF + 0));
    if (kHasB) {
        s_block(dQb, dk0, tS_b);
        mma_commit(bar(B_SF + 1));
    }
    mma_commit(bar(B_KE + st.ks));
    next_k();
    // tiles 1 .. n_kv-1
    uint32_t acc0 = 0u;
    for (int j = 1; j < n_kv; ++j) {
        tile((st.pa + (uint32_t)j - 1u) & 1u, (st.pb + (uint32_t)j - 1u) & 1u, acc0, wait_oe && j == 1);
        acc0 = 1u;
        next_k();
        next_v();
    }
    mma_commit(bar(B_QF));    // every S of the pair issued: Q is free once they complete
    // last P.V pair: P_x(n_kv - 1) with V tile n_kv - 1
    const uint64_t dvl = dV0 + (uint64_t)st.vs * kTileDesc;
    wait(B_PF + 0, (st.pa + (uint32_t)n_kv - 1u) & 1u);
    wait(B_VF + st.vs, st.vph);
    if (wait_oe && n_kv == 1) wait(B_OE, oe_par);
    pv_block(tS_a, dvl, tO_a, acc0);
    if (kHasB) {
        wait(B_PF + 1, (st.pb + (uint32_t)n_kv - 1u) & 1u);
        pv_block(tS_b, dvl, tO_b, acc0);
    }
    mma_commit(bar(B_VE + st.vs));
    next_v();
    mma_commit(bar(B_OD));
    st.pa += (uint32_t)n_kv;
    if (kHasB) st.pb += (uint32_t)n_kv;
}

// The MMA issuer for a pair with one query tile (tile A) and n_kv >= 2 key tiles, the key tiles
// split between the two halves of TMEM: tiles 0, 2, 4, ... go to (S_A, O_A), tiles 1, 3, 5, ...
// to (S_B, O_B), and the two softmax warpgroups each run an online softmax over their half, so
// that one half's softmax overlaps the other's MMAs as two query tiles' do (warpgroup A merges
// the halves at the end).  Issue order: S(0), S(1), then per key tile j: P(j).V(j), S(j + 2)
// on the same half (in issue order after the P.V that reads the P it overwrites).
__device__ __forceinline__ void mma_issuer_kpp(const TcParams& P, uint32_t tmem, uint32_t sQ, uint32_t sK,
                                               uint32_t sV, uint32_t sBar, int n_kv, int q_ready,
                                               uint32_t q_par, RingState& st, bool wait_oe, uint32_t oe_par,
                                               volatile uint32_t* abort) {
    auto bar = [&](int i) { return sBar + 8u * (uint32_t)i; };
    constexpr uint32_t idS = idesc_bf16(BM, BN, false);
    constexpr uint32_t idO = idesc_bf16(BM, HD, true);
    constexpr uint64_t kTileDesc = (uint64_t)(TILE >> 4);
    const uint64_t dQa = sw128_desc(sQ, 16, 1024);
    const uint64_t dK0 = sw128_desc(sK, 16, 1024);
    const uint64_t dV0 = sw128_desc(sV, HALF_TILE, 1024);
    const uint32_t tS_a = tmem + kColS, tS_b = tmem + kColS + BN;
    const uint32_t tO_a = tmem + kColO, tO_b = tmem + kColO + HD;
    auto wait = [&](int i, uint32_t parity) {
        mbar_wait(bar(i), parity, P.err, abort);
        tc_fence_after();
    };
    int ks = st.ks, vs = st.vs;
    uint32_t kph = st.kph, vph = st.vph;
    auto s_next = [&](int x) {        // S of the next key tile into half x, its K stage released after
        wait(B_KF + ks, kph);
        const uint64_t dk = dK0 + (uint64_t)ks * kTileDesc;
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk) {
            const uint64_t off = (uint64_t)(((kk >> 2) * HALF_TILE + (kk & 3) * 32) >> 4);
            mma_bf16(x ? tS_b : tS_a, dQa + off, dk + off, idS, kk > 0 ? 1u : 0u);
        }
        mma_commit(bar(B_SF + x));
        mma_commit(bar(B_KE + ks));
        kph ^= ks == KSTAGES - 1 ? 1u : 0u;
        ks = ks == KSTAGES - 1 ? 0 : ks + 1;
    };
    wait(q_ready, q_par);
    s_next(0);
    s_next(1);
    uint32_t pa = st.pa, pb = st.pb;   // P phases of each half completed before this pair
#pragma unroll 1
    for (int j = 0; j < n_kv; ++j) {
        const int x = j & 1;
        wait(B_PF + x, (x ? pb : pa) & 1u);
        pa += x ? 0u : 1u;
        pb += x ? 1u : 0u;
        wait(B_VF + vs, vph);
        if (wait_oe && j == 0) wait(B_OE, oe_par);
        const uint64_t dv = dV0 + (uint64_t)vs * kTileDesc;
#pragma unroll
        for (int kk = 0; kk < BN / 16; ++kk)
            mma_bf16_ts(x ? tO_b : tO_a, (x ? tS_b : tS_a) + (uint32_t)kk * 8u,
                        dv + (uint64_t)((kk * 2048) >> 4), idO, kk > 0 || j >= 2 ? 1u : 0u);
        mma_commit(bar(B_VE + vs));
        vph ^= vs == VSTAGES - 1 ? 1u : 0u;
        vs = vs == VSTAGES - 1 ? 0 : vs + 1;
        if (j + 2 < n_kv) s_next(x);
    }
    mma_commit(bar(B_QF));
    mma_commit(bar(B_OD));
    st.ks = ks;
    st.kph = kph;
    st.vs = vs;
    st.vph = vph;
    st.pa = pa;
    st.pb = pb;
}

// ------------------------------------------------------------------ fused loaders

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}
// generic-proxy writes to shared memory become visible to the tensor core's (async) reads
__device__ __forceinline__ void fence_proxy_async() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ uint4 lds128(uint32_t a) {
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "r"(a)
                 : "memory");
    return v;
}
__device__ __forceinline__ void sts128(uint32_t a, const uint4& v) {
    asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(a), "r"(v.x), "r"(v.y), "r"(v.z),
                 "r"(v.w)
                 : "memory");
}
// Byte offset of 16-byte chunk q (0..7) of row r in a 128-row, 128-byte-wide swizzled block
// (the SWIZZLE_128B layout: the chunk index XOR the row index mod 8).
__device__ __forceinline__ uint32_t sw_off(int r, int q) {
    return (uint32_t)(r * 128 + ((q ^ (r & 7)) << 4));
}

// A walk over one request's occurrences in composed-row order.  The occurrence table sits
// in the kernel parameters; a dependent chain of reads there costs a memory latency per
// step, so each walk keeps its current occurrence in registers and reads the table only
// when a row moves past it (rows only increase).
struct OccWalk {
    int idx;    // current occurrence
    int beg;    // its first composed row (relative to the request)
    int end;    // one past its last
    int src;    // pool slot of row beg
};
__device__ __forceinline__ void walk_load(OccWalk& w, const FusedTcParams& F, int i) {
    w.idx = i;
    w.beg = F.occ[i].dest_row;
    w.end = w.beg + F.occ[i].m;
    w.src = F.occ[i].src_row;
}
__device__ __forceinline__ void walk_to(OccWalk& w, const FusedTcParams& F, int R, int o_end) {
    while (R >= w.end && w.idx + 1 < o_end) walk_load(w, F, w.idx + 1);
}
// Pool slot of composed slot row R, or -1 (bounds-check bit set) if it is out of range.
__device__ __forceinline__ int64_t walk_slot(OccWalk& w, const FusedTcParams& F, int R, int o_end) {
    walk_to(w, F, R, o_end);
    const int64_t slot = (int64_t)w.src + (R - w.beg);
    if (R < w.beg || R >= w.end || slot < 0 || slot >= F.pool_slots) {
        atomicOr(F.t.err, 1);
        return -1;
    }
    return slot;
}
// Whether the 8-row group of composed row R (rows R & ~7 .. +7) is not one contiguous run of
// one source: several occurrences, composed slots and suffix rows, or rows past the suffix
// (`used` = slots + suffix tokens; those rows are zeros).  Clean groups are moved by TMA,
// ragged ones row by row.
__device__ __forceinline__ bool group_ragged(OccWalk& w, const FusedTcParams& F, int R, int n_slots,
                                            int used, int o_end) {
    const int gs = R & ~7, ge = gs + 8;
    if (R >= n_slots) return gs < n_slots || ge > used;
    walk_to(w, F, R, o_end);
    return !(w.beg <= gs && ge <= w.end);
}

// The fused kernel's TMA producer (one thread): for each key tile, K and V each as soon as
// their stage is free.  A tile from one source (a single occurrence's pool slots, or 128 of
// the request's suffix rows) is two 128-row boxes; a mixed tile is moved as runs of clean
// 8-row groups in boxes of 64 and 8 rows (its ragged groups are left to the loaders).  The
// stage's "landed" barrier expects the bytes of the boxes issued.  Suffix rows of V come from
// v_suf; those of K are copied by the K loaders from the cache, where the softmax warps
// write them turned (generic-proxy stores, which TMA would need a proxy fence to see).
__device__ __forceinline__ void fused_producer(const FusedTcParams& F, int l, int bl, int hk, int j_base,
                                               int n_kv, bool writer, uint32_t sK, uint32_t sV,
                                               uint32_t sBar, volatile uint32_t* abort) {
    const TcParams& P = F.t;
    auto bar = [&](int i) { return sBar + 8u * (uint32_t)i; };
    const int lg = P.layer0 + l;
    const int n_slots = P.req[bl].n_slots;
    const int used = n_slots + P.sq;
    const int o_begin = F.req_occ[bl];
    const int o_end = F.req_occ[bl + 1];
    const int pool_row0 = (int)((int64_t)lg * F.pool_slots);
    // suffix row R (R >= n_slots) of V: row sfx_row0 + R of v_suf
    const int sfx_row0 = (l * P.batch_total + P.b0 + bl) * P.sq - n_slots;
    OccWalk wk{}, wv{};
    if (o_end > o_begin) {
        walk_load(wk, F, o_begin);
        wv = wk;
    }
    auto tile = [&](int jt, bool is_v, OccWalk& w, uint32_t dst, uint32_t landed) {
        const CUtensorMap* pool128 = is_v ? &F.tm_pv : &F.tm_pk;
        const CUtensorMap* pool8 = is_v ? &F.tm_pv8 : &F.tm_pk8;
        const int R0 = (j_base + jt) * BN;
        if (is_v && R0 >= n_slots && R0 + BN <= used) {      // 128 suffix rows of V
            mbar_expect_tx(landed, TILE);
            tma_load_3d(dst, &F.tm_sv, 0, hk, sfx_row0 + R0, landed);
            tma_load_3d(dst + HALF_TILE, &F.tm_sv, 64, hk, sfx_row0 + R0, landed);
            return;
        }
        if (R0 < n_slots) {
            walk_to(w, F, R0, o_end);
            if (w.beg <= R0 && R0 + BN <= w.end && (int64_t)w.src + (R0 - w.beg) + BN <= F.pool_slots &&
                w.src + (R0 - w.beg) >= 0) {                  // one occurrence
                const int row = pool_row0 + w.src + (R0 - w.beg);
                mbar_expect_tx(landed, TILE);
                tma_load_3d(dst, pool128, 0, hk, row, landed);
                tma_load_3d(dst + HALF_TILE, pool128, 64, hk, row, landed);
                return;
            }
        }
        // mixed: runs of clean groups whose source rows are contiguous, each moved in boxes of
        // 64 and 8 rows; the bytes are counted in a first walk, the boxes issued in a second
        const CUtensorMap* pool64 = is_v ? &F.tm_pv64 : &F.tm_pk64;
        auto runs = [&](OccWalk& wr, bool issue) -> int {
            int groups = 0;
            int g0 = -1, ng = 0, row0 = 0;
            bool sfx0 = false;
            auto flush = [&]() {
                if (ng == 0) return;
                groups += ng;
                if (issue) {
                    int g = g0, left = ng;
                    while (left > 0) {
                        const bool big = left >= 8;
                        const int n = big ? 8 : 1;
                        const CUtensorMap* tm = sfx0 ? (big ? &F.tm_sv64 : &F.tm_sv8) : (big ? pool64 : pool8);
                        const int row = row0 + 8 * (g - g0);
                        const uint32_t d = dst + (uint32_t)g * 1024u;
                        tma_load_3d(d, tm, 0, hk, row, landed);
                        tma_load_3d(d + HALF_TILE, tm, 64, hk, row, landed);
                        g += n;
                        left -= n;
                    }
                }
                ng = 0;
            };
            for (int g = 0; g < BN / 8; ++g) {
                const int R = R0 + 8 * g;
                const bool is_sfx = R >= n_slots;
                bool clean = !group_ragged(wr, F, R, n_slots, used, o_end) && (is_v || !is_sfx);
                int row = 0;
                if (clean) {
                    if (is_sfx) {
                        row = sfx_row0 + R;
                    } else {
                        const int64_t slot = (int64_t)wr.src + (R - wr.beg);
                        clean = slot >= 0 && slot + 8 <= F.pool_slots;   // else the loaders report it
                        row = pool_row0 + (int)slot;
                    }
                }
                if (!clean) {
                    flush();
                    continue;
                }
                if (ng > 0 && is_sfx == sfx0 && row == row0 + 8 * ng) {
                    ++ng;                                     // the run goes on
                } else {
                    flush();
                    g0 = g;
                    ng = 1;
                    row0 = row;
                    sfx0 = is_sfx;
                }
            }
            flush();
            return groups;
        };
        OccWalk w2 = w;
        const int clean = runs(w2, false);
        mbar_expect_tx(landed, (uint32_t)clean * 8u * 256u);
        runs(w, true);
    };
    // a stage is free once the MMA has read it and, in the CTAs that store the composed
    // rows, once the store of its tile to the cache has read it too (non-blocking tests: the
    // producer serves whichever ring frees a stage first)
    auto k_free = [&](int j) {
        const uint32_t ph = (uint32_t)((j / KSTAGES) - 1) & 1u;
        return j < KSTAGES || (mbar_test(bar(B_KE + j % KSTAGES), ph) &&
                               (!writer || mbar_test(bar(B_KW + j % KSTAGES), ph)));
    };
    auto v_free = [&](int j) {
        const uint32_t ph = (uint32_t)((j / VSTAGES) - 1) & 1u;
        return j < VSTAGES || (mbar_test(bar(B_VE + j % VSTAGES), ph) &&
                               (!writer || mbar_test(bar(B_VW + j % VSTAGES), ph)));
    };
    int jk = 0, jv = 0;
    long long idle0 = -1;      // start of the current wait for a free stage
    while (jk < n_kv || jv < n_kv) {
        if (jk < n_kv && k_free(jk)) {
            const int st = jk % KSTAGES;
            tile(jk, false, wk, sK + (uint32_t)(st * TILE), bar(B_KL + st));
            ++jk;
            idle0 = -1;
            continue;
        }
        if (jv < n_kv && v_free(jv)) {
            const int st = jv % VSTAGES;
            tile(jv, true, wv, sV + (uint32_t)(st * TILE), bar(B_VL + st));
            ++jv;
            idle0 = -1;
            continue;
        }
        // nothing issuable: poll both rings again, within the wait limit
        if (*abort) return;
        const long long now = clock64();
        if (idle0 < 0) {
            idle0 = now;
        } else if (now - idle0 > kWaitCycles) {
            atomicOr(P.err, 2);
            *abort = 1u;
            return;
        }
    }
}

// The fused kernel's producer after the CTA's first pair, when the CTA runs the pairs of its
// (layer, request, KV head) in turn: the first was the last pair, which composed the whole
// cache; pairs 0 .. pairs - 2 follow and read it.  Each pair's Q tiles (before RoPE) once the
// previous pair's S MMAs have read the last ones; the K and V tiles whole from the cache once
// the writer's stores are complete (B_WD), each as its stage frees (a stage last used by a
// first-pair tile is free once its store has read it too).  n_first: the first pair's tiles.
__device__ __noinline__ void fused_rest_producer(const FusedTcParams& F, int l, int bl, int b, int hk,
                                                    int p_count, int s_r, int n_first, uint32_t sQ,
                                                    uint32_t sK, uint32_t sV, uint32_t sBar,
                                                    volatile uint32_t* abort) {
    const TcParams& P = F.t;
    auto bar = [&](int i) { return sBar + 8u * (uint32_t)i; };
    const int G = P.group;
    const int qz = l * P.batch_total + b;
    const int key0 = (int)((int64_t)(P.layer0 + l) * P.rows + P.req[bl].row_base);
    // the CTA's pair pi >= 1 is pair pi - 1 of the request
    int qi = 1;
    int pk = 1, jk = 0, gk = n_first;
    int pv = 1, jv = 0, gv = n_first;
    PairSpan sk = pair_span(P, 0, 0, s_r), sv = sk;
    bool stored = false;
    auto k_free = [&](int g) {
        const uint32_t ph = (uint32_t)((g / KSTAGES) - 1) & 1u;
        return g < KSTAGES || (mbar_test(bar(B_KE + g % KSTAGES), ph) &&
                               (g - KSTAGES >= n_first || mbar_test(bar(B_KW + g % KSTAGES), ph)));
    };
    auto v_free = [&](int g) {
        const uint32_t ph = (uint32_t)((g / VSTAGES) - 1) & 1u;
        return g < VSTAGES || (mbar_test(bar(B_VE + g % VSTAGES), ph) &&
                               (g - VSTAGES >= n_first || mbar_test(bar(B_VW + g % VSTAGES), ph)));
    };
    long long idle0 = -1;
    while (qi < p_count || pk < p_count || pv < p_count) {
        if (!stored) stored = mbar_test(bar(B_WD), 0u);
        if (qi < p_count && mbar_test(bar(B_QF), (uint32_t)(qi - 1) & 1u)) {
            const PairSpan sq = pair_span(P, qi - 1, 0, s_r);
            mbar_expect_tx(bar(B_Q), sq.has_b ? 2 * TILE : TILE);
            tma_load_4d(sQ, &P.tm_q, 0, hk * G, sq.t0a, qz, bar(B_Q));
            tma_load_4d(sQ + HALF_TILE, &P.tm_q, 64, hk * G, sq.t0a, qz, bar(B_Q));
            if (sq.has_b) {
                tma_load_4d(sQ + TILE, &P.tm_q, 0, hk * G, sq.t0b, qz, bar(B_Q));
                tma_load_4d(sQ + TILE + HALF_TILE, &P.tm_q, 64, hk * G, sq.t0b, qz, bar(B_Q));
            }
            ++qi;
            idle0 = -1;
            continue;
        }
        if (stored && pk < p_count && k_free(gk)) {
            const int st = gk % KSTAGES;
            const int row = key0 + (sk.j_base + jk) * BN;
            mbar_expect_tx(bar(B_KL + st), TILE);
            tma_load_3d(sK + (uint32_t)(st * TILE), &P.tm_k, 0, hk, row, bar(B_KL + st));
            tma_load_3d(sK + (uint32_t)(st * TILE) + HALF_TILE, &P.tm_k, 64, hk, row, bar(B_KL + st));
            ++gk;
            if (++jk == sk.n_kv) {
                jk = 0;
                if (++pk < p_count) sk = pair_span(P, pk - 1, 0, s_r);
            }
            idle0 = -1;
            continue;
        }
        if (stored && pv < p_count && v_free(gv)) {
            const int st = gv % VSTAGES;
            const int row = key0 + (sv.j_base + jv) * BN;
            mbar_expect_tx(bar(B_VL + st), TILE);
            tma_load_3d(sV + (uint32_t)(st * TILE), &P.tm_v, 0, hk, row, bar(B_VL + st));
            tma_load_3d(sV + (uint32_t)(st * TILE) + HALF_TILE, &P.tm_v, 64, hk, row, bar(B_VL + st));
            ++gv;
            if (++jv == sv.n_kv) {
                jv = 0;
                if (++pv < p_count) sv = pair_span(P, pv - 1, 0, s_r);
            }
            idle0 = -1;
            continue;
        }
        if (*abort) return;
        const long long now = clock64();
        if (idle0 < 0) {
            idle0 = now;
        } else if (now - idle0 > kWaitCycles) {
            atomicOr(P.err, 2);
            *abort = 1u;
            return;
        }
    }
}

__device__ __forceinline__ void tma_store_3d(const CUtensorMap* tm, uint32_t src, int c0, int c1, int c2) {
    asm volatile("cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%1, %2, %3}], [%4];" ::"l"(
                     reinterpret_cast<uint64_t>(tm)),
                 "r"(c0), "r"(c1), "r"(c2), "r"(src)
                 : "memory");
}

// Store a whole 128-row tile (two 64-channel halves) of a stage to the cache by TMA, as one
// bulk async-group (the caller waits for its read of shared memory before freeing the stage).
__device__ __forceinline__ void issue_store(const CUtensorMap* tm, uint32_t src, int hk, int row) {
    tma_store_3d(tm, src, 0, hk, row);
    tma_store_3d(tm, src + HALF_TILE, 64, hk, row);
    asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}

// Two pairs turned at once on the packed fp32 pipe: per lane exactly rotate1 (the product
// rounded, then a fused multiply-add).  x, y: the pairs' two channels; c, s: their cos, sin.
__device__ __forceinline__ void rotate2(float2 x, float2 y, float2 c, float2 s, float2& ox, float2& oy) {
    asm("{\n\t.reg .b64 px, py, pc, ps, t, u, a, b;\n\t"
        "mov.b64 px, {%4, %5};\n\t"
        "mov.b64 py, {%6, %7};\n\t"
        "mov.b64 pc, {%8, %9};\n\t"
        "mov.b64 ps, {%10, %11};\n\t"
        "mul.rn.f32x2 t, py, ps;\n\t"
        "xor.b64 t, t, 0x8000000080000000;\n\t"
        "fma.rn.f32x2 a, px, pc, t;\n\t"
        "mul.rn.f32x2 u, py, pc;\n\t"
        "fma.rn.f32x2 b, px, ps, u;\n\t"
        "mov.b64 {%0, %1}, a;\n\t"
        "mov.b64 {%2, %3}, b;\n\t}"
        : "=f"(ox.x), "=f"(ox.y), "=f"(oy.x), "=f"(oy.y)
        : "f"(x.x), "f"(x.y), "f"(y.x), "f"(y.y), "f"(c.x), "f"(c.y), "f"(s.x), "f"(s.y));
}

// bf16 pair <-> fp32 pair
__device__ __forceinline__ float2 bf2_to_f2(uint32_t w) {
    return make_float2(__uint_as_float(w << 16), __uint_as_float(w & 0xffff0000u));
}
__device__ __forceinline__ uint32_t f2_to_bf2(float lo, float hi) {
    __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&h);
}

// The K loaders of the fused kernel (warps 12..15, lt = 0..127).  Per key tile, thread lt
// owns chunk pair kc = lt % 8 (channels 8kc.. and 64+8kc..) of rows lt/8 + 16i: it copies
// the ragged rows among them (cp.async, 16 bytes a chunk, into the swizzled layout TMA
// produces; suffix rows from the cache, once the softmax warps have turned them) and zeroes
// those past the suffix, waits for the tile's TMA part, turns its chunks of composed slots
// by their occurrence's offset (the writer CTAs in layer 0, KV head 0 also write the slots'
// positions), and releases the stage to the MMA and the writer.  They wait only for a K
// stage to be free, so they run up to two tiles ahead of the MMA.
__device__ __forceinline__ void fused_k_loader(const FusedTcParams& F, int lt, int l, int bl, int hk,
                                               bool writer, int j_base, int n_kv, int n_all, uint32_t sK,
                                               uint8_t* gK, uint32_t sBar, volatile uint32_t* abort) {
    using bf = __nv_bfloat16;
    const TcParams& P = F.t;
    auto bar = [&](int i) { return sBar + 8u * (uint32_t)i; };
    const int lg = P.layer0 + l;
    const ReqParam& rq = P.req[bl];
    const int n_slots = rq.n_slots;
    const int used = n_slots + P.sq;
    const int row_base = rq.row_base;
    const int o_begin = F.req_occ[bl];
    const int o_end = F.req_occ[bl + 1];
    const int64_t hkv = P.hkv;
    const int64_t pool_row0 = (int64_t)lg * F.pool_slots;
    const int64_t cache_row0 = (int64_t)lg * P.rows + row_base;
    const bf* pk = static_cast<const bf*>(F.pool_k);
    const bf* ck = static_cast<const bf*>(F.cache_k);
    const int kc = lt & 7, kr0 = lt >> 3;
    const bool pos_writer = writer && lg == 0 && hk == 0 && kc == 0;
    OccWalk wk{}, wr{};
    if (o_end > o_begin) {
        walk_load(wk, F, o_begin);
        wr = wk;
    }
    float2* occ_cs = F.occ_cs + (int64_t)l * F.n_occ * 64;    // this layer's table
    int cs_occ = -1;          // occurrence whose angles cc, ss hold
    bool k_turned = false;    // the suffix rows' K' are in the cache
    float2 cc[4], ss[4];      // cos and sin of this thread's 8 frequencies, in pairs
    auto load_cs = [&](int idx) {
        const float4* t = reinterpret_cast<const float4*>(occ_cs + idx * 64 + 8 * kc);
#pragma unroll
        for (int w = 0; w < 4; ++w) {
            const float4 v = t[w];                     // (cos, sin) of two frequencies
            cc[w] = make_float2(v.x, v.z);
            ss[w] = make_float2(v.y, v.w);
        }
        cs_occ = idx;
    };
    // chunk pair (x, y) of a row turned by cc, ss
    auto turn_pair = [&](const uint4& xa, const uint4& ya, uint4& xo, uint4& yo) {
        const uint32_t xw[4] = {xa.x, xa.y, xa.z, xa.w}, yw[4] = {ya.x, ya.y, ya.z, ya.w};
        uint32_t a[4], b[4];
#pragma unroll
        for (int w = 0; w < 4; ++w) {
            float2 gx, gy;
            rotate2(bf2_to_f2(xw[w]), bf2_to_f2(yw[w]), cc[w], ss[w], gx, gy);
            a[w] = f2_to_bf2(gx.x, gx.y);
            b[w] = f2_to_bf2(gy.x, gy.y);
        }
        xo = make_uint4(a[0], a[1], a[2], a[3]);
        yo = make_uint4(b[0], b[1], b[2], b[3]);
    };
    // (cos, sin) of the request's occurrences at the 64 frequencies, evaluated while the
    // first tiles are on their way into this layer's rows of the scratch table (the CTAs of
    // the layer and request write the same values; a table per layer keeps the CTAs that
    // write one line few) and read back as a row per occurrence while turning
    {
        const uint64_t turn = F.rope.turn[lt & 63];     // entry e has frequency e % 64 = lt % 64
        for (int e = (o_begin << 6) + lt; e < (o_end << 6); e += kLoaders)
            occ_cs[e] = turn_cs(turn, F.occ[e >> 6].delta);
    }
    asm volatile("bar.sync 1, %0;" ::"n"(kLoaders) : "memory");

    for (int jt = 0; jt < n_kv; ++jt) {
        const int R0 = (j_base + jt) * BN;
        const int st_i = jt % KSTAGES;
        const uint32_t st = sK + (uint32_t)(st_i * TILE);
        if (jt >= KSTAGES)    // stage free: S_A and S_B of tile jt - KSTAGES finished
            mbar_wait(bar(B_KE + st_i), (uint32_t)((jt / KSTAGES) - 1) & 1u, P.err, abort);
        // a tile of one occurrence (the producer moves it whole): no ragged row, one set of
        // angles, loaded while the tile lands
        bool whole = false;
        if (R0 + BN <= n_slots && o_end > o_begin) {
            walk_to(wk, F, R0, o_end);
            const int64_t s0 = (int64_t)wk.src + (R0 - wk.beg);
            whole = wk.beg <= R0 && R0 + BN <= wk.end && s0 >= 0 && s0 + BN <= F.pool_slots;
        }
#pragma unroll 1
        for (int i = 0; i < (whole ? 0 : BN / 16); ++i) {
            const int r = kr0 + 16 * i;
            const int R = R0 + r;
            if (R < n_slots && !group_ragged(wk, F, R, n_slots, used, o_end)) continue;
            if (R >= used) {                              // past the suffix: zeros
                sts128(st + sw_off(r, kc), make_uint4(0u, 0u, 0u, 0u));
                sts128(st + HALF_TILE + sw_off(r, kc), make_uint4(0u, 0u, 0u, 0u));
                continue;
            }
            const bf* src;
            if (R < n_slots) {
                const int64_t slot = walk_slot(wk, F, R, o_end);
                if (slot < 0) continue;
                src = pk + ((pool_row0 + slot) * hkv + hk) * HD;
            } else {
                if (!k_turned) {
                    mbar_wait(bar(B_SK), 0u, P.err, abort);
                    k_turned = true;
                }
                src = ck + ((cache_row0 + R) * hkv + hk) * HD;
            }
            cp_async16(st + sw_off(r, kc), src + 8 * kc);
            cp_async16(st + HALF_TILE + sw_off(r, kc), src + 64 + 8 * kc);
        }
        cp_async_commit();
        if (whole) {
            wr = wk;
            if (wr.idx != cs_occ) load_cs(wr.idx);
        }
        cp_async_wait<0>();
        mbar_wait(bar(B_KL + st_i), (uint32_t)(jt / KSTAGES) & 1u, P.err, abort);
        if (whole) {
            // two rows at a time, plain shared-memory accesses, so that the loads of both
            // rows are in flight together
            uint8_t* g = gK + st_i * TILE;
#pragma unroll 1
            for (int i = 0; i < BN / 16; i += 2) {
                uint4* p0 = reinterpret_cast<uint4*>(g + sw_off(kr0 + 16 * i, kc));
                uint4* p1 = reinterpret_cast<uint4*>(g + sw_off(kr0 + 16 * i + 16, kc));
                constexpr int kY = HALF_TILE / 16;             // the partner channels' block
                const uint4 x0 = p0[0], y0 = p0[kY], x1 = p1[0], y1 = p1[kY];
                uint4 a0, b0, a1, b1;
                turn_pair(x0, y0, a0, b0);
                turn_pair(x1, y1, a1, b1);
                p0[0] = a0;
                p0[kY] = b0;
                p1[0] = a1;
                p1[kY] = b1;
            }
            if (pos_writer) {
                const FusedOcc& o = F.occ[wr.idx];
#pragma unroll 1
                for (int i = 0; i < BN / 16; ++i) {
                    const int R = R0 + kr0 + 16 * i;
                    F.pos[row_base + R] = o.delta + min((R - o.dest_row + 1) * o.k, o.n) - 1;
                }
            }
        } else {
#pragma unroll 1
            for (int i = 0; i < BN / 16; ++i) {
                const int r = kr0 + 16 * i;
                const int R = R0 + r;
                if (R >= n_slots) break;                       // suffix rows are already turned
                if (walk_slot(wr, F, R, o_end) < 0) continue;
                if (wr.idx != cs_occ) load_cs(wr.idx);
                const uint32_t a0 = st + sw_off(r, kc);
                uint4 xo, yo;
                turn_pair(lds128(a0), lds128(a0 + HALF_TILE), xo, yo);
                sts128(a0, xo);
                sts128(a0 + HALF_TILE, yo);
                if (pos_writer) {
                    const FusedOcc& o = F.occ[wr.idx];
                    F.pos[row_base + R] = o.delta + min((R - o.dest_row + 1) * o.k, o.n) - 1;
                }
            }
        }
        fence_proxy_async();
        mbar_arrive(bar(B_KF + st_i));
    }
    // the key tiles of the CTA's later pairs (pairs run in turn) come whole from the composed
    // cache: passed on to the MMA as they land
    for (int g = n_kv; g < n_all; ++g) {
        const int st_i = g % KSTAGES;
        mbar_wait(bar(B_KL + st_i), (uint32_t)(g / KSTAGES) & 1u, P.err, abort);
        mbar_arrive(bar(B_KF + st_i));
    }
}

// The writer of the fused kernel (warp 2, one thread, writer CTAs): once the loaders have
// released a tile, its K' (composed slots and suffix rows turned, zero rows past the suffix)
// and its V go to the cache by TMA; both stores are in flight together, and each stage is
// handed back to the producer as soon as its store has read it.
__device__ __forceinline__ void fused_writer(const FusedTcParams& F, int l, int bl, int hk, int j_base,
                                             int n_kv, uint32_t sK, uint32_t sV, uint32_t sBar,
                                             bool more_pairs, volatile uint32_t* abort) {
    const TcParams& P = F.t;
    auto bar = [&](int i) { return sBar + 8u * (uint32_t)i; };
    const int cache_row0 = (int)((int64_t)(P.layer0 + l) * P.rows + P.req[bl].row_base);
    for (int jt = 0; jt < n_kv; ++jt) {
        const int R0 = (j_base + jt) * BN;
        const int ks = jt % KSTAGES, vs = jt % VSTAGES;
        mbar_wait(bar(B_KF + ks), (uint32_t)(jt / KSTAGES) & 1u, P.err, abort);
        issue_store(&P.tm_k, sK + (uint32_t)(ks * TILE), hk, cache_row0 + R0);
        mbar_wait(bar(B_VF + vs), (uint32_t)(jt / VSTAGES) & 1u, P.err, abort);
        issue_store(&P.tm_v, sV + (uint32_t)(vs * TILE), hk, cache_row0 + R0);
        asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory");    // K's store read
        mbar_arrive(bar(B_KW + ks));
        asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");    // V's
        mbar_arrive(bar(B_VW + vs));
    }
    if (more_pairs) {
        asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
        mbar_arrive(bar(B_WD));     // the composed cache is written: later pairs may read it
    }
    // otherwise nothing in this CTA reads the cache back: the stores have read shared memory
    // (above), and their writes complete with the grid
}

// The V loader of the fused kernel (warp 3, lt = 0..31): per key tile, the ragged 8-row
// groups' rows by cp.async, or zeros past the suffix (thread lt: chunk lt % 16 of rows
// lt/16 + 2u of each such group), then the tile's TMA part, then the stage is released to
// the MMA and the writer.
__device__ __forceinline__ void fused_v_loader(const FusedTcParams& F, int lt, int l, int bl, int hk,
                                               int j_base, int n_kv, int n_all, uint32_t sV, uint32_t sBar,
                                               volatile uint32_t* abort) {
    using bf = __nv_bfloat16;
    const TcParams& P = F.t;
    auto bar = [&](int i) { return sBar + 8u * (uint32_t)i; };
    const int lg = P.layer0 + l;
    const int n_slots = P.req[bl].n_slots;
    const int used = n_slots + P.sq;
    const int o_begin = F.req_occ[bl];
    const int o_end = F.req_occ[bl + 1];
    const int64_t hkv = P.hkv;
    const int64_t pool_row0 = (int64_t)lg * F.pool_slots;
    const int64_t sfx_row0 = ((int64_t)l * P.batch_total + P.b0 + bl) * P.sq - n_slots;
    const bf* pv = static_cast<const bf*>(F.pool_v);
    const bf* sv = static_cast<const bf*>(F.v_suf);
    const int vq = lt & 15, vr0 = lt >> 4;
    OccWalk wv{};
    if (o_end > o_begin) walk_load(wv, F, o_begin);
    for (int jt = 0; jt < n_kv; ++jt) {
        const int R0 = (j_base + jt) * BN;
        const int st_i = jt % VSTAGES;
        const uint32_t st = sV + (uint32_t)(st_i * TILE) + (uint32_t)((vq >> 3) * HALF_TILE);
        if (jt >= VSTAGES)    // stage free: both P.V of tile jt - VSTAGES finished
            mbar_wait(bar(B_VE + st_i), (uint32_t)((jt / VSTAGES) - 1) & 1u, P.err, abort);
#pragma unroll 1
        for (int g = 0; g < BN / 8; ++g) {
            if (!group_ragged(wv, F, R0 + 8 * g, n_slots, used, o_end)) continue;
#pragma unroll 1
            for (int u = 0; u < 4; ++u) {
                const int r = 8 * g + vr0 + 2 * u;
                const int R = R0 + r;
                if (R >= used) {                          // past the suffix: zeros
                    sts128(st + sw_off(r, vq & 7), make_uint4(0u, 0u, 0u, 0u));
                    continue;
                }
                const bf* src;
                if (R < n_slots) {
                    const int64_t slot = walk_slot(wv, F, R, o_end);
                    if (slot < 0) continue;
                    src = pv + ((pool_row0 + slot) * hkv + hk) * HD;
                } else {
                    src = sv + ((sfx_row0 + R) * hkv + hk) * HD;
                }
                cp_async16(st + sw_off(r, vq & 7), src + 8 * vq);
            }
        }
        cp_async_commit();
        cp_async_wait<0>();
        mbar_wait(bar(B_VL + st_i), (uint32_t)(jt / VSTAGES) & 1u, P.err, abort);
        fence_proxy_async();
        mbar_arrive(bar(B_VF + st_i));
    }
    for (int g = n_kv; g < n_all; ++g) {     // the later pairs' tiles, whole from the cache
        const int st_i = g % VSTAGES;
        mbar_wait(bar(B_VL + st_i), (uint32_t)(g / VSTAGES) & 1u, P.err, abort);
        mbar_arrive(bar(B_VF + st_i));
    }
}

// The suffix preparation of the fused kernel, done by the softmax warps (ts = 0..255) while
// they wait for their first S tile.  Item (token tt, chunk pair q = ts % 8) takes the angles
// of position L_r + tt at the 8 frequencies of chunk pair q (from the table that
// suffix_angles_kernel evaluates once per launch) and turns with them
//   - chunk pair q of the G query rows of token tt in shared memory, for tt in [q_lo, q_hi)
//     (this CTA's query tokens), once Q has landed; then the MMA issuer is told (B_QR);
//   - chunk pair q of suffix row tt's K, from k_suf into the cache, for tt in [k_lo, k_hi)
//     (the suffix rows among this CTA's key tiles; the CTAs of a request write the same
//     bits), with the row's position in the CTAs that own the positions; then the K loaders,
//     which copy these rows into the K tiles, are told (B_SK).
// The K rows of a thread's first two items are loaded before anything else and their angles
// kept from the query pass, so the query rows, which the first MMA waits for, go first.  The
// angles (turn_cs) and the rounding are the suffix kernel's.
__device__ __forceinline__ void fused_suffix_prep(const FusedTcParams& F, int ts, int l, int bl, int hk,
                                                  int k_lo, int k_hi, int q_lo, int q_hi, bool pos_rows,
                                                  uint32_t q_par, bool first, uint32_t sQ, uint32_t sBar,
                                                  volatile uint32_t* abort) {
    using bf = __nv_bfloat16;
    const TcParams& P = F.t;
    auto bar = [&](int i) { return sBar + 8u * (uint32_t)i; };
    const ReqParam& rq = P.req[bl];
    const int64_t pos0 = (int64_t)rq.l_req + rq.t0;
    const int G = P.group, tq = P.tq;
    const int q = ts & 7;                  // every item of this thread has chunk pair q
    const float2* tab = F.sfx_cs + (int64_t)bl * P.sq * 64 + 8 * q;
    const int64_t row_elems = (int64_t)P.hkv * HD;
    const bf* ksrc = static_cast<const bf*>(F.k_suf) +
                     ((int64_t)l * P.batch_total + P.b0 + bl) * P.sq * row_elems + hk * HD + 8 * q;
    bf* kdst = static_cast<bf*>(F.cache_k) +
               ((int64_t)(P.layer0 + l) * P.rows + rq.row_base + rq.n_slots) * row_elems + hk * HD + 8 * q;
    int lo = 0, hi = 0;
    if (k_hi > k_lo) {
        lo = k_lo;
        hi = k_hi;
    }
    if (q_hi > q_lo) {
        lo = hi > lo ? min(lo, q_lo) : q_lo;
        hi = max(hi, q_hi);
    }
    const int n_items = (hi - lo) * 8;     // item i: token lo + i / 8, chunk pair i % 8
    // (cos, sin) of token tt at chunk pair q's 8 frequencies, from the table of the grid
    // launched before this one (read from L2)
    auto angles = [&](int tt, float2 (&cc)[4], float2 (&ss)[4]) {
        const float4* t = reinterpret_cast<const float4*>(tab + (int64_t)tt * 64);
#pragma unroll
        for (int w = 0; w < 4; ++w) {
            const float4 v = __ldcg(t + w);
            cc[w] = make_float2(v.x, v.z);
            ss[w] = make_float2(v.y, v.w);
        }
    };
    auto turn_chunks = [&](const uint4& xv, const uint4& yv, const float2 (&cc)[4], const float2 (&ss)[4],
                           uint4& xo, uint4& yo) {
        const uint32_t xw[4] = {xv.x, xv.y, xv.z, xv.w}, yw[4] = {yv.x, yv.y, yv.z, yv.w};
        uint32_t a[4], b[4];
#pragma unroll
        for (int w = 0; w < 4; ++w) {
            float2 gx, gy;
            rotate2(bf2_to_f2(xw[w]), bf2_to_f2(yw[w]), cc[w], ss[w], gx, gy);
            a[w] = f2_to_bf2(gx.x, gx.y);
            b[w] = f2_to_bf2(gy.x, gy.y);
        }
        xo = make_uint4(a[0], a[1], a[2], a[3]);
        yo = make_uint4(b[0], b[1], b[2], b[3]);
    };
    auto is_k = [&](int tt) { return tt >= k_lo && tt < k_hi; };
    auto is_q = [&](int tt) { return tt >= q_lo && tt < q_hi; };
    bool q_landed = false;
    auto q_item = [&](int tt, const float2 (&cc)[4], const float2 (&ss)[4]) {
        if (!q_landed) {
            mbar_wait(bar(B_Q), q_par, P.err, abort);
            q_landed = true;
        }
        const int x = (tt - q_lo) / tq;           // tile A or B
        const int t = tt - q_lo - x * tq;         // token within the tile
        const uint32_t base = sQ + (uint32_t)x * TILE;
#pragma unroll 1
        for (int g = 0; g < G; ++g) {
            const uint32_t a0 = base + sw_off(t * G + g, q);
            uint4 xo, yo;
            turn_chunks(lds128(a0), lds128(a0 + HALF_TILE), cc, ss, xo, yo);
            sts128(a0, xo);
            sts128(a0 + HALF_TILE, yo);
        }
    };
    auto k_item = [&](int tt, const uint4& xa, const uint4& ya, const float2 (&cc)[4],
                      const float2 (&ss)[4]) {
        uint4 xo, yo;
        turn_chunks(xa, ya, cc, ss, xo, yo);
        st16(kdst + tt * row_elems, xo);
        st16(kdst + tt * row_elems + 64, yo);
        if (pos_rows && q == 0) F.pos[rq.row_base + rq.n_slots + tt] = (int32_t)(pos0 + tt);
    };
    // the first two items: their K rows are loaded first and stay in flight while the query
    // rows are turned, and their angles are kept for the K pass
    const int t_0 = lo + (ts >> 3), t_1 = t_0 + 32;
    const bool v0 = ts < n_items, v1 = ts + 256 < n_items;
    const bool k0 = v0 && is_k(t_0), k1 = v1 && is_k(t_1);
    uint4 x0 = make_uint4(0u, 0u, 0u, 0u), y0 = x0, x1 = x0, y1 = x0;
    if (k0) {
        x0 = ld16(ksrc + t_0 * row_elems);
        y0 = ld16(ksrc + t_0 * row_elems + 64);
    }
    if (k1) {
        x1 = ld16(ksrc + t_1 * row_elems);
        y1 = ld16(ksrc + t_1 * row_elems + 64);
    }
    float2 c0[4], s0[4], c1[4], s1[4];
    // the table's grid has finished and its writes are visible (returns at once when this
    // grid was launched after it completed)
    if (n_items > 0) asm volatile("griddepcontrol.wait;" ::: "memory");
    // both items' angles in flight before either is used
    if (v0) angles(t_0, c0, s0);
    if (v1) angles(t_1, c1, s1);
    if (v0 && is_q(t_0)) q_item(t_0, c0, s0);
    if (v1 && is_q(t_1)) q_item(t_1, c1, s1);
#pragma unroll 1
    for (int i = ts + 512; i < n_items; i += 256) {
        const int tt = lo + (i >> 3);
        if (!is_q(tt)) continue;
        float2 cc[4], ss[4];
        angles(tt, cc, ss);
        q_item(tt, cc, ss);
    }
    fence_proxy_async();
    mbar_arrive(bar(B_QR));
    if (k0) k_item(t_0, x0, y0, c0, s0);
    if (k1) k_item(t_1, x1, y1, c1, s1);
#pragma unroll 1
    for (int i = ts + 512; i < n_items; i += 256) {
        const int tt = lo + (i >> 3);
        if (!is_k(tt)) continue;
        const uint4 xa = ld16(ksrc + tt * row_elems), ya = ld16(ksrc + tt * row_elems + 64);
        float2 cc[4], ss[4];
        angles(tt, cc, ss);
        k_item(tt, xa, ya, cc, ss);
    }
    if (first) mbar_arrive(bar(B_SK));    // the K loaders read these rows with cp.async
}

// The plain kernel's TMA producer (one thread) for the pairs [p_first, p_first + p_count)
// that its CTA runs in turn: a pair's Q tiles once the MMAs of the previous pair have read
// the last ones (B_QF), and the pairs' K and V tiles in order, each as soon as its ring stage
// is free; whichever of the three can go first goes.
template <bool kSif>
__device__ __forceinline__ void plain_producer(const TcParams& P, int l, int bl, int b, int hk,
                                               int p_first, int p_count, int sp, int s_r, uint32_t sQ,
                                               uint32_t sK, uint32_t sV, uint32_t sBar,
                                               volatile uint32_t* abort) {
    auto bar = [&](int i) { return sBar + 8u * (uint32_t)i; };
    const int G = P.group;
    const int qz = l * P.batch_total + b;
    const int key0 = (int)((int64_t)(P.layer0 + l) * P.rows + P.req[bl].row_base);
    // launched as a programmatic dependent: the grid before it (which wrote Q and the newest
    // key rows) has completed and its writes are visible (returns at once otherwise)
    asm volatile("griddepcontrol.wait;" ::: "memory");
    int qi = 0;                             // next pair whose Q tiles to load
    int pk = 0, jk = 0, gk = 0;             // K: pair, tile within it, tiles issued in all
    int pv = 0, jv = 0, gv = 0;             // V: the same
    PairSpan sk = pair_span(P, p_first, sp, s_r), sv = sk;
    long long idle0 = -1;                   // start of the current wait for a free stage
    while (qi < p_count || pk < p_count || pv < p_count) {
        if (qi < p_count && (qi == 0 || mbar_test(bar(B_QF), (uint32_t)(qi - 1) & 1u))) {
            const PairSpan sq = pair_span(P, p_first + qi, sp, s_r);
            mbar_expect_tx(bar(B_Q), sq.has_b ? 2 * TILE : TILE);
            tma_load_4d(sQ, &P.tm_q, 0, hk * G, sq.t0a, qz, bar(B_Q));
            tma_load_4d(sQ + HALF_TILE, &P.tm_q, 64, hk * G, sq.t0a, qz, bar(B_Q));
            if (sq.has_b) {
                tma_load_4d(sQ + TILE, &P.tm_q, 0, hk * G, sq.t0b, qz, bar(B_Q));
                tma_load_4d(sQ + TILE + HALF_TILE, &P.tm_q, 64, hk * G, sq.t0b, qz, bar(B_Q));
            }
            ++qi;
            idle0 = -1;
            continue;
        }
        if (pk < p_count && (gk < KSTAGES || mbar_test(bar(B_KE + gk % KSTAGES),
                                                       (uint32_t)((gk / KSTAGES) - 1) & 1u))) {
            const int s = gk % KSTAGES;
            const int krow = key0 + (kSif ? span_tile(sk, jk) : sk.j_base + jk) * BN;
            mbar_expect_tx(bar(B_KF + s), TILE);
            tma_load_3d(sK + s * TILE, &P.tm_k, 0, hk, krow, bar(B_KF + s));
            tma_load_3d(sK + s * TILE + HALF_TILE, &P.tm_k, 64, hk, krow, bar(B_KF + s));
            ++gk;
            if (++jk == sk.n_kv) {
                jk = 0;
                if (++pk < p_count) sk = pair_span(P, p_first + pk, sp, s_r);
            }
            idle0 = -1;
            continue;
        }
        if (pv < p_count && (gv < VSTAGES || mbar_test(bar(B_VE + gv % VSTAGES),
                                                       (uint32_t)((gv / VSTAGES) - 1) & 1u))) {
            const int s = gv % VSTAGES;
            const int vrow = key0 + (kSif ? span_tile(sv, jv) : sv.j_base + jv) * BN;
            mbar_expect_tx(bar(B_VF + s), TILE);
            tma_load_3d(sV + s * TILE, &P.tm_v, 0, hk, vrow, bar(B_VF + s));
            tma_load_3d(sV + s * TILE + HALF_TILE, &P.tm_v, 64, hk, vrow, bar(B_VF + s));
            ++gv;
            if (++jv == sv.n_kv) {
                jv = 0;
                if (++pv < p_count) sv = pair_span(P, p_first + pv, sp, s_r);
            }
            idle0 = -1;
            continue;
        }
        // nothing issuable: poll again, within the wait limit
        if (*abort) return;
        const long long now = clock64();
        if (idle0 < 0) {
            idle0 = now;
        } else if (now - idle0 > kWaitCycles) {
            atomicOr(P.err, 2);
            *abort = 1u;
            return;
        }
    }
}

// The table of the suffix tokens' (cos, sin) at the 64 frequencies, [B][Sq][64], evaluated once
// per fused launch (turn_cs, as the suffix kernel evaluates them) rather than by each of the
// request's CTAs.  It lets the dependent fused grid start at once (programmatic dependent
// launch): only the fused kernel's softmax warps wait for it, the pool loads and the K
// rotation do not.
struct SfxAngles {
    float2* tab;
    int32_t sq, batch;
    RopeTurns rope;
    ReqParam req[kMaxFusedReq];
};
__global__ void __launch_bounds__(256) suffix_angles_kernel(const __grid_constant__ SfxAngles A) {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    const int64_t n = (int64_t)A.batch * A.sq * 64;
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < n; e += (int64_t)gridDim.x * blockDim.x) {
        const int64_t bt = e >> 6;                       // request * Sq + token
        const int b = (int)(bt / A.sq);
        const int tt = (int)(bt - (int64_t)b * A.sq);
        A.tab[e] = turn_cs(A.rope.turn[e & 63], (int64_t)A.req[b].l_req + A.req[b].t0 + tt);
    }
}

// kFused: compose + suffix preparation + attention; kMulti (fused only): the CTA runs every
// pair of query tiles of its (layer, request, KV head), the last pair first (it composes the
// cache), the others from the cache.  A separate instantiation, so that the one-pair fused
// kernel keeps its register allocation.  kSif (plain only): extraction C2 rows
// (TcParams::sif_k), a kernel of its own (attn_tc_sif_kernel) so that the plain kernel's code
// stays as it is.
template <bool kFused, bool kMulti, bool kSif, bool kKpp = false>
__device__ __forceinline__ void attn_tc_body(const typename KernelParams<kFused>::type& KP) {
    const TcParams& P = tc_params(KP);
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~uintptr_t(1023));
    const uint32_t sQ = smem_u32(smem);             // Q_A, then Q_B
    const uint32_t sK = sQ + 2 * TILE;
    const uint32_t sV = sK + KSTAGES * TILE;
    const uint32_t sBar = sV + VSTAGES * TILE;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + (size_t)TILE * kSmemTiles + 8 * NBAR);
    volatile uint32_t* abort = tmem_slot + 1;      // set by the first wait that gives up
    auto bar = [&](int i) { return sBar + 8u * (uint32_t)i; };

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int G = P.group;
    const int hk = blockIdx.y;
    const int l = blockIdx.z / P.batch;
    const int bl = blockIdx.z - l * P.batch;
    const int b = P.b0 + bl;
    const int s_r = P.req[bl].n_slots + P.req[bl].t0;   // keys before the first query token
    // pairs of Q tiles: the CTA runs pairs [p_first, p_first + p_count) in turn (one pair
    // unless the plain kernel groups short pairs); the groups go last first: under a causal
    // mask the later pairs see more keys, so the longest CTAs start in the first wave
    const int n_groups = (int)(gridDim.x / P.n_split);
    const int p_first = (n_groups - 1 - (int)(blockIdx.x / P.n_split)) * P.pair_group;
    const int p_count = min(P.pairs, p_first + P.pair_group) - p_first;
    const int sp = (int)(blockIdx.x % P.n_split);   // key-range split
    // the pair the CTA runs first: its first one, except in a fused CTA that runs every pair of
    // its (layer, request, KV head), where the last pair leads (see fused_rest_producer)
    const int p_lead = (kMulti && p_count > 1) ? P.pairs - 1 : p_first;
    // fused: the CTAs of the last pair see every key row of the request (all of the suffix),
    // so they write the composed cache
    const bool writer = p_lead == P.pairs - 1;
    const PairSpan ps0 = pair_span(P, p_lead, sp, s_r);
    // key tiles of all the CTA's pairs (the fused loaders pass the later pairs' tiles on)
    int n_all = ps0.n_kv;
    if (kMulti && p_count > 1)
        for (int pr = 0; pr < P.pairs - 1; ++pr) n_all += pair_span(P, pr, sp, s_r).n_kv;
    const int t0a = ps0.t0a;
    const int t0b = ps0.t0b;
    const bool has_b = ps0.has_b;
    const int j_base = ps0.j_base;
    const int n_kv = ps0.n_kv;

    if (!kFused && threadIdx.x == 0 && n_kv > 0) {
        // the first pair's Q tiles and first key tile on their way into L2 while the CTA sets
        // up (barriers, TMEM, register split), so that the producer's first loads find them
        // there (llama8b attention 59.7 -> 58.4 us, a 2187-key decode step 32.8 -> 31.2 us;
        // the same for the fused kernel's first pool tile gained nothing)
        const int qz = l * P.batch_total + b;
        const int key0 = (int)((int64_t)(P.layer0 + l) * P.rows + P.req[bl].row_base);
        const int row = key0 + (kSif ? span_tile(ps0, 0) : j_base) * BN;
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            tma_prefetch_4d(&P.tm_q, 64 * h, hk * G, t0a, qz);
            if (has_b) tma_prefetch_4d(&P.tm_q, 64 * h, hk * G, t0b, qz);
            tma_prefetch_3d(&P.tm_k, 64 * h, hk, row);
            tma_prefetch_3d(&P.tm_v, 64 * h, hk, row);
        }
    }
    if (threadIdx.x == 0) {
        mbar_init(bar(B_Q), 1);
        // a full stage is one TMA arrival (with its byte count), or every loader's arrival
        for (int s = 0; s < KSTAGES; ++s) {
            mbar_init(bar(B_KF + s), kFused ? (uint32_t)kLoaders : 1u);
            mbar_init(bar(B_KE + s), 1);
        }
        for (int s = 0; s < VSTAGES; ++s) {
            mbar_init(bar(B_VF + s), kFused ? (uint32_t)kVLoaders : 1u);
            mbar_init(bar(B_VE + s), 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(bar(B_SF + i), 1);
            mbar_init(bar(B_PF + i), 128);
        }
        for (int s = 0; s < KSTAGES; ++s) {
            mbar_init(bar(B_KL + s), 1);
            mbar_init(bar(B_KW + s), 1);
        }
        for (int s = 0; s < VSTAGES; ++s) {
            mbar_init(bar(B_VL + s), 1);
            mbar_init(bar(B_VW + s), 1);
        }
        mbar_init(bar(B_QR), 256u);
        mbar_init(bar(B_SK), 256u);
        mbar_init(bar(B_QF), 1u);
        mbar_init(bar(B_OE), 256u);
        mbar_init(bar(B_WD), 1u);
        mbar_init(bar(B_OD), 1);
        *abort = 0u;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         smem_u32(tmem_slot)),
                     "r"(kTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    // a programmatic dependent launched after this grid (the split merge) may start now: it
    // waits for this grid before it reads what this one writes
    if (!kFused && threadIdx.x == 0) asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

    if (warp < 4) {
        asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(kFused ? kRegsLowFused : kRegsLow));
        if (warp == 0 && lane == 0 && n_kv > 0) {
            // ------------------------------------------------------------ TMA producer
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&P.tm_q)) : "memory");
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&P.tm_k)) : "memory");
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&P.tm_v)) : "memory");
            if constexpr (kFused) {
                const int qz = l * P.batch_total + b;
                mbar_expect_tx(bar(B_Q), has_b ? 2 * TILE : TILE);
                tma_load_4d(sQ, &P.tm_q, 0, hk * G, t0a, qz, bar(B_Q));
                tma_load_4d(sQ + HALF_TILE, &P.tm_q, 64, hk * G, t0a, qz, bar(B_Q));
                if (has_b) {
                    tma_load_4d(sQ + TILE, &P.tm_q, 0, hk * G, t0b, qz, bar(B_Q));
                    tma_load_4d(sQ + TILE + HALF_TILE, &P.tm_q, 64, hk * G, t0b, qz, bar(B_Q));
                }
                fused_producer(KP, l, bl, hk, j_base, n_kv, writer, sK, sV, sBar, abort);
                if constexpr (kMulti)
                    if (p_count > 1)
                        fused_rest_producer(KP, l, bl, b, hk, p_count, s_r, n_kv, sQ, sK, sV, sBar, abort);
            } else {
                plain_producer<kSif>(P, l, bl, b, hk, p_first, p_count, sp, s_r, sQ, sK, sV, sBar, abort);
            }
        } else if (warp == 1 && lane == 0 && n_kv > 0) {
            // ------------------------------------------------------------ MMA issuer
            RingState st;
            if constexpr (kFused && !kMulti) {   // one pair
                if (has_b)
                    mma_issuer<true>(P, tmem, sQ, sK, sV, sBar, n_kv, B_QR, 0u, st, false, 0u, abort);
                else
                    mma_issuer<false>(P, tmem, sQ, sK, sV, sBar, n_kv, B_QR, 0u, st, false, 0u, abort);
            } else if constexpr (kFused) {       // the lead pair, then pairs 0 .. pairs - 2
                for (int pi = 0; pi < p_count; ++pi) {
                    const PairSpan ps = pi == 0 ? ps0 : pair_span(P, pi - 1, sp, s_r);
                    const uint32_t q_par = (uint32_t)pi & 1u, oe_par = (uint32_t)(pi - 1) & 1u;
                    if (ps.has_b)
                        mma_issuer<true>(P, tmem, sQ, sK, sV, sBar, ps.n_kv, B_QR, q_par, st, pi > 0, oe_par, abort);
                    else
                        mma_issuer<false>(P, tmem, sQ, sK, sV, sBar, ps.n_kv, B_QR, q_par, st, pi > 0, oe_par, abort);
                }
            } else {
                for (int pi = 0; pi < p_count; ++pi) {
                    const PairSpan ps = pi == 0 ? ps0 : pair_span(P, p_first + pi, sp, s_r);
                    const uint32_t q_par = (uint32_t)pi & 1u, oe_par = (uint32_t)(pi - 1) & 1u;
                    if (ps.has_b)
                        mma_issuer<true>(P, tmem, sQ, sK, sV, sBar, ps.n_kv, B_Q, q_par, st, pi > 0, oe_par, abort);
                    else if (kKpp && ps.n_kv >= 2 && pi == p_count - 1)   // key tiles ping-pong
                        mma_issuer_kpp(P, tmem, sQ, sK, sV, sBar, ps.n_kv, B_Q, q_par, st, pi > 0, oe_par, abort);
                    else
                        mma_issuer<false>(P, tmem, sQ, sK, sV, sBar, ps.n_kv, B_Q, q_par, st, pi > 0, oe_par, abort);
                }
            }
        } else if (warp == 2 && lane == 0 && n_kv > 0 && writer) {
            // ------------------------------------------------------------ writer (fused)
            if constexpr (kFused)
                fused_writer(KP, l, bl, hk, j_base, n_kv, sK, sV, sBar, kMulti && p_count > 1, abort);
        } else if (warp == 3 && n_kv > 0) {
            // ------------------------------------------------------------ V loader (fused)
            if constexpr (kFused)
                fused_v_loader(KP, lane, l, bl, hk, j_base, n_kv, kMulti ? n_all : n_kv, sV, sBar, abort);
        }
    } else if (warp < 12) {
        asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(kFused ? kRegsHighFused : kRegsHigh));
        // ---------------------------------------------------------------- softmax warps
        const int x = warp >= 8 ? 1 : 0;               // tile A (warps 4..7) or B (8..11)
        if constexpr (kFused && !kMulti) {
            // the suffix rows among this CTA's key tiles, and its query tokens
            const int k_lo = max(0, j_base * BN - s_r);
            const int k_hi = min(P.sq, (j_base + n_kv) * BN - s_r);
            const int q_hi = n_kv > 0 ? ps0.t_last + 1 : t0a;   // (the loaders run iff n_kv > 0)
            fused_suffix_prep(KP, (int)threadIdx.x - 128, l, bl, hk, k_lo, k_hi, t0a, q_hi,
                              writer && P.layer0 + l == 0 && hk == 0, 0u, true, sQ, sBar, abort);
            if (x == 0 || has_b)
                softmax_tile<false>(P, tmem, sBar, x, warp & 3, lane, x ? t0b : t0a, l, bl, b, hk, sp, ps0,
                             0u, 0u, false, abort, sQ);
        } else if constexpr (kFused) {
            // per pair: the suffix preparation (the lead pair's also turns the suffix rows
            // among its key tiles into the cache), then the softmax over its key tiles
            uint32_t done = 0u;
            for (int pi = 0; pi < p_count; ++pi) {
                const PairSpan ps = pi == 0 ? ps0 : pair_span(P, pi - 1, sp, s_r);
                const int k_lo = pi == 0 ? max(0, ps.j_base * BN - s_r) : 0;
                const int k_hi = pi == 0 ? min(P.sq, (ps.j_base + ps.n_kv) * BN - s_r) : 0;
                const int q_hi = ps.n_kv > 0 ? ps.t_last + 1 : ps.t0a;   // (the loaders run iff n_kv > 0)
                fused_suffix_prep(KP, (int)threadIdx.x - 128, l, bl, hk, k_lo, k_hi, ps.t0a, q_hi,
                                  pi == 0 && writer && P.layer0 + l == 0 && hk == 0, (uint32_t)pi & 1u,
                                  pi == 0, sQ, sBar, abort);
                if (x == 0 || ps.has_b) {
                    softmax_tile<false>(P, tmem, sBar, x, warp & 3, lane, x ? ps.t0b : ps.t0a, l, bl, b, hk, sp,
                                 ps, done, (uint32_t)pi & 1u, p_count > 1, abort,
                                 pi == p_count - 1 ? sQ : 0u);
                    done += (uint32_t)ps.n_kv;
                } else if (p_count > 1) {
                    mbar_arrive(bar(B_OE));
                }
            }
        } else {
            uint32_t done = 0u;     // S_x tiles of the earlier pairs
            for (int pi = 0; pi < p_count; ++pi) {
                const PairSpan ps = pi == 0 ? ps0 : pair_span(P, p_first + pi, sp, s_r);
                // one query tile over two or more key tiles (the CTA's last pair): the two
                // warpgroups take alternate key tiles (mma_issuer_kpp) and merge at the end
                const bool kpp = kKpp && !ps.has_b && ps.n_kv >= 2 && pi == p_count - 1;
                if (x == 0 || ps.has_b || kpp) {
                    softmax_tile<true, kSif, kKpp>(P, tmem, sBar, x, warp & 3, lane, x && !kpp ? ps.t0b : ps.t0a, l, bl,
                                 b, hk, sp, ps, done, (uint32_t)pi & 1u, p_count > 1, abort,
                                 pi == p_count - 1 ? sQ : 0u, kpp);
                    done += kpp ? (uint32_t)((ps.n_kv + 1 - x) / 2) : (uint32_t)ps.n_kv;
                } else if (p_count > 1) {    // no tile B in this pair: nothing of O to read
                    mbar_arrive(bar(B_OE));
                } else if (P.tickets != nullptr) {   // a split without tile B: the merge's two
                    asm volatile("bar.sync 4, 256;" ::: "memory");   // barriers (no rows, no
                    asm volatile("bar.sync 4, 256;" ::: "memory");   // ticket of its own)
                }
            }
        }
    } else {
        if constexpr (kFused) {
            asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(kRegsLoadFused));
            // ------------------------------------------------------------ loaders (fused)
            if (n_kv > 0)
                fused_k_loader(KP, (int)threadIdx.x - 12 * 32, l, bl, hk, writer, j_base, n_kv,
                               kMulti ? n_all : n_kv, sK, smem + 2 * TILE, sBar, abort);
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                     "r"(kTmemCols)
                     : "memory");
    }
}

template <bool kFused, bool kMulti = false>
__global__ void __launch_bounds__(kFused ? kThreadsFused : kThreads, 1)
    attn_tc_kernel(const __grid_constant__ typename KernelParams<kFused>::type KP) {
    attn_tc_body<kFused, kMulti, false>(KP);
}

__global__ void __launch_bounds__(kThreads, 1) attn_tc_sif_kernel(const __grid_constant__ TcParams KP) {
    attn_tc_body<false, false, true>(KP);
}

// Decode steps (AttnParams::key_pingpong): the plain kernel whose last pair, when it has one
// query tile, splits its key tiles between the two softmax warpgroups.
__global__ void __launch_bounds__(kThreads, 1) attn_tc_decode_kernel(const __grid_constant__ TcParams KP) {
    attn_tc_body<false, false, false, true>(KP);
}

// The kernel of an instantiation.
template <bool kFused, bool kMulti, bool kSif, bool kKpp = false>
const void* tc_kernel_fn() {
    if constexpr (kSif) return reinterpret_cast<const void*>(&attn_tc_sif_kernel);
    else if constexpr (kKpp) return reinterpret_cast<const void*>(&attn_tc_decode_kernel);
    else return reinterpret_cast<const void*>(&attn_tc_kernel<kFused, kMulti>);
}

// Merge the splits: lse = log2 sum_s 2^lse_s, O = sum_s 2^(lse_s - lse) O_s.  One warp per
// (layer, request, suffix token, query head) row; lane i owns head channels 4i .. 4i+3.
// Every split's lse and O slice is loaded before any is used (at most kMaxSplit), so the
// loads of one row are all in flight together.
constexpr int kMaxSplit = 16;

__global__ void __launch_bounds__(256) attn_combine_kernel(const __grid_constant__ AttnParams P) {
    asm volatile("griddepcontrol.wait;" ::: "memory");   // the partials are complete and visible
    const int64_t rows = (int64_t)P.lq * P.batch_total * P.sq * P.hq;
    const int64_t row = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (row >= rows) return;
    const int h = (int)(row % P.hq);
    const int64_t lbt = row / P.hq;                 // (l * Btot + b) * Sq + t
    const int t = (int)(lbt % P.sq);
    const int64_t lb = lbt / P.sq;
    const int64_t lse_id = (lb * P.hq + h) * P.sq + t;
    float ls[kMaxSplit];
    float4 o[kMaxSplit];
#pragma unroll
    for (int s = 0; s < kMaxSplit; ++s) {
        ls[s] = -CUDART_INF_F;
        o[s] = make_float4(0.f, 0.f, 0.f, 0.f);
        if (s < P.n_split) {
            ls[s] = P.part_lse[(int64_t)s * rows + lse_id];
            o[s] = *reinterpret_cast<const float4*>(P.part_o + ((int64_t)s * rows + row) * HD + lane * 4);
        }
    }
    float mx = -CUDART_INF_F;
#pragma unroll
    for (int s = 0; s < kMaxSplit; ++s) mx = fmaxf(mx, ls[s]);
    float wsum = 0.f;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int s = 0; s < kMaxSplit; ++s) {
        const float w = ls[s] == -CUDART_INF_F ? 0.f : ex2(ls[s] - mx);
        acc.x += w * o[s].x;
        acc.y += w * o[s].y;
        acc.z += w * o[s].z;
        acc.w += w * o[s].w;
        wsum += w;
    }
    const float inv = 1.0f / wsum;
    uint2 pk;
    pk.x = pack_bf16(acc.x * inv, acc.y * inv);
    pk.y = pack_bf16(acc.z * inv, acc.w * inv);
    *reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(P.out) + row * HD + lane * 4) = pk;
    if (P.lse != nullptr && lane == 0) P.lse[lse_id] = (mx + log2f(wsum)) * 0.69314718055994531f;
}

// ------------------------------------------------------------------ host side

bool encode(CUtensorMap* tm, const void* base, int rank, const cuuint64_t* dims,
            const cuuint64_t* strides_bytes, const cuuint32_t* box) {
    return encode_tensor_map(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, rank, base, dims, strides_bytes,
                             box, CU_TENSOR_MAP_SWIZZLE_128B);
}

}  // namespace

bool encode_tensor_map(CUtensorMap* tm, CUtensorMapDataType type, int rank, const void* base,
                       const cuuint64_t* dims, const cuuint64_t* strides_bytes, const cuuint32_t* box,
                       CUtensorMapSwizzle swizzle) {
    // the driver entry point, looked up once (a function-local static: thread-safe)
    static const PFN_cuTensorMapEncodeTiled_v12000 fn = []() -> PFN_cuTensorMapEncodeTiled_v12000 {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q{};
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
        return nullptr;
    }();
    if (!fn) return false;
    cuuint32_t estr[5] = {1, 1, 1, 1, 1};
    const CUresult r = fn(tm, type, (cuuint32_t)rank, const_cast<void*>(base), dims, strides_bytes, box,
                          estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle,
                          CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

int64_t attn_tc_units(int hq, int hkv, int sq, int lq, int batch) {
    const int tq = BM / (hq / hkv);
    const int64_t tiles = (sq + tq - 1) / tq;
    return (tiles + 1) / 2 * hkv * lq * batch;     // one CTA per pair of query tiles
}

cudaError_t launch_attn_combine(const AttnParams& a, cudaStream_t s) {
    (void)cudaGetLastError();
    if (a.n_split > kMaxSplit || (a.sq_pitch != 0 && a.sq_pitch != a.sq)) return cudaErrorInvalidValue;
    const int64_t rows = (int64_t)a.lq * a.batch_total * a.sq * a.hq;
    const int64_t blocks = (rows + 7) / 8;
    if (blocks > 0x7fffffffLL) return cudaErrorInvalidValue;
    if (a.dependent) {          // its launch overlaps the attention's last CTAs
        cudaLaunchConfig_t cfg{};
        cfg.gridDim = dim3((unsigned)blocks);
        cfg.blockDim = dim3(256);
        cfg.stream = s;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        const cudaError_t e = cudaLaunchKernelEx(&cfg, attn_combine_kernel, a);
        if (e != cudaSuccess) return e;
    } else {
        attn_combine_kernel<<<(unsigned)blocks, 256, 0, s>>>(a);
    }
    return cudaGetLastError();
}

bool attn_tc_supported(int dtype, int d, int hq, int hkv) {
    if (dtype != kDtypeBf16 || d != HD || hkv < 1 || hq % hkv) return false;
    const int g = hq / hkv;
    return g == 1 || g == 2 || g == 4 || g == 8 || g == 16;
}

namespace {

// Host-side preparation shared by the plain and the fused launch: function attributes once
// per process, the register-split guard, the tensor maps and the scalar parameters.
template <bool kFused, bool kMulti = false, bool kSif = false, bool kKpp = false>
cudaError_t prepare_tc(const AttnParams& a, TcParams& p, dim3& grid) {
    constexpr int threads = kFused ? kThreadsFused : kThreads;
    constexpr int high = kFused ? kRegsHighFused : kRegsHigh;
    constexpr int low_total = kFused ? 128 * (kRegsLowFused + kRegsLoadFused) : 128 * kRegsLow;
    // once per process (one device per context; function-local statics: thread-safe)
    static const cudaError_t smem_err = cudaFuncSetAttribute(
        tc_kernel_fn<kFused, kMulti, kSif, kKpp>(), cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes);
    if (smem_err != cudaSuccess) return smem_err;
    {   // the register split must not ask for more than the launch holds
        static const int launch_regs = []() {
            cudaFuncAttributes fa{};
            return cudaFuncGetAttributes(&fa, tc_kernel_fn<kFused, kMulti, kSif, kKpp>()) == cudaSuccess ? fa.numRegs : -1;
        }();
        if (launch_regs < 0) return cudaErrorInvalidDeviceFunction;
        if (launch_regs * threads < low_total + 256 * high) return cudaErrorInvalidConfiguration;
    }
    const int pitch = a.sq_pitch > 0 ? a.sq_pitch : a.sq;
    if (pitch < a.sq || (pitch != a.sq && a.n_split > 1)) return cudaErrorInvalidValue;
    std::memset(&p, 0, sizeof(p));
    const int G = a.hq / a.hkv;
    const int tq = BM / G;
    {   // Q: q_rot [Lq*Btot][Sq'][Hq][128] -> dims (d, Hq, Sq, Lq*Btot); tokens past Sq read 0
        const cuuint64_t dims[4] = {HD, (cuuint64_t)a.hq, (cuuint64_t)a.sq,
                                    (cuuint64_t)a.lq * a.batch_total};
        const cuuint64_t str[3] = {(cuuint64_t)HD * 2, (cuuint64_t)a.hq * HD * 2,
                                   (cuuint64_t)pitch * a.hq * HD * 2};
        const cuuint32_t box[4] = {64, (cuuint32_t)G, (cuuint32_t)tq, 1};
        if (!encode(&p.tm_q, a.q_rot, 4, dims, str, box)) return cudaErrorInvalidValue;
        // out has q's layout: its 128-row tiles leave through the same boxes
        if (!encode(&p.tm_o, a.out, 4, dims, str, box)) return cudaErrorInvalidValue;
    }
    {   // K, V: cache [L*rows][Hkv][128] -> dims (d, Hkv, L*rows); layer0 + lq <= L
        const int64_t lrows = (int64_t)(a.layer0 + a.lq) * a.rows;
        const cuuint64_t dims[3] = {HD, (cuuint64_t)a.hkv, (cuuint64_t)lrows};
        const cuuint64_t str[2] = {(cuuint64_t)HD * 2, (cuuint64_t)a.hkv * HD * 2};
        const cuuint32_t box[3] = {64, 1, (cuuint32_t)BN};
        if (!encode(&p.tm_k, a.cache_k, 3, dims, str, box)) return cudaErrorInvalidValue;
        if (!encode(&p.tm_v, a.cache_v, 3, dims, str, box)) return cudaErrorInvalidValue;
    }
    p.out = a.out;
    p.lse = a.lse;
    p.err = a.err;
    p.rows = a.rows;
    p.layer0 = a.layer0;
    p.lq = a.lq;
    p.batch = a.batch;
    p.batch_total = a.batch_total;
    p.b0 = a.b0;
    p.sq = a.sq;
    p.sq_pitch = pitch;
    p.hq = a.hq;
    p.hkv = a.hkv;
    p.group = G;
    p.tq = tq;
    p.scale_log2 = a.scale_log2;
    p.n_split = a.n_split < 1 ? 1 : a.n_split;
    p.part_o = a.part_o;
    p.part_lse = a.part_lse;
    p.tickets = kFused || p.n_split == 1 || p.n_split > kMaxMergeSplits ? nullptr : a.tickets;
    p.sif_k = a.sif_k;

    if (kSif != (a.sif_k > 0) || a.sif_k < 0 || (kSif && (kFused || p.n_split != 1))) return cudaErrorInvalidValue;
    if (kKpp != (a.key_pingpong != 0) || (kKpp && (kFused || kSif))) return cudaErrorInvalidValue;
    if (a.batch < 1 || a.batch > kMaxReq) return cudaErrorInvalidValue;
    std::memcpy(p.req, a.req, sizeof(ReqParam) * (size_t)a.batch);
    const int64_t pairs = ((a.sq + tq - 1) / tq + 1) / 2;
    // The plain kernel runs several pairs of one (layer, request, KV head) per CTA when the
    // launch is many waves of CTAs: each CTA's fixed cost (TMEM, barriers, the first tiles
    // from HBM, the epilogue) is then paid once for several short pairs (causal extraction
    // rows: 1 to 4 key tiles a pair).  The context's attn_pairs setting caps the choice.
    int64_t pg = 1;
    if (kMulti) {                // every pair of a (layer, request, KV head) in one CTA
        if (p.n_split != 1) return cudaErrorInvalidValue;
        pg = pairs;
    } else if (!kFused && p.n_split == 1) {
        static const int sms = []() {
            int dev = 0, n = 0;
            if (cudaGetDevice(&dev) != cudaSuccess ||
                cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 1)
                return 1;
            return n;
        }();
        const int64_t ctas = pairs * a.hkv * a.lq * a.batch;
        pg = std::max<int64_t>(1, std::min<int64_t>(pairs, ctas / sms));
        if (a.pairs_per_cta >= 1) pg = std::min<int64_t>(pairs, a.pairs_per_cta);
    }
    p.pairs = (int32_t)pairs;
    p.pair_group = (int32_t)pg;
    const int64_t gx = (pairs + pg - 1) / pg * p.n_split;
    if (gx > 0x7fffffffLL) return cudaErrorInvalidValue;
    grid = dim3((unsigned)gx, a.hkv, a.lq * a.batch);
    if (grid.z > 65535u || grid.y > 65535u) return cudaErrorInvalidValue;
    return cudaSuccess;
}

}  // namespace

cudaError_t preload_attn_tc_kernels() {
    cudaFuncAttributes fa{};
    return cudaFuncGetAttributes(&fa, attn_tc_kernel<false>);
}

cudaError_t launch_attn_tc(const AttnParams& a, cudaStream_t s, Hook before) {
    (void)cudaGetLastError();   // report this launch's error only, not a stale one
    TcParams p;
    dim3 grid;
    if (a.sif_k > 0) {          // extraction C2 rows: their own instantiation, launched plainly
        cudaError_t e = prepare_tc<false, false, true>(a, p, grid);
        if (e != cudaSuccess) return e;
        before();
        attn_tc_sif_kernel<<<grid, kThreads, kSmemBytes, s>>>(p);
        return cudaGetLastError();
    }
    cudaError_t e = a.key_pingpong ? prepare_tc<false, false, false, true>(a, p, grid) : prepare_tc<false>(a, p, grid);
    if (e != cudaSuccess) return e;
    before();
    if (a.dependent) {          // starts while the kernel before it runs (the producer waits)
        cudaLaunchConfig_t cfg{};
        cfg.gridDim = grid;
        cfg.blockDim = dim3(kThreads);
        cfg.dynamicSmemBytes = kSmemBytes;
        cfg.stream = s;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        e = a.key_pingpong ? cudaLaunchKernelEx(&cfg, attn_tc_decode_kernel, p)
                           : cudaLaunchKernelEx(&cfg, attn_tc_kernel<false>, p);
        if (e != cudaSuccess) return e;
    } else if (a.key_pingpong) {
        attn_tc_decode_kernel<<<grid, kThreads, kSmemBytes, s>>>(p);
    } else {
        attn_tc_kernel<false><<<grid, kThreads, kSmemBytes, s>>>(p);
    }
    return cudaGetLastError();
}

namespace {
thread_local FusedTcParams g_fused;          // the prepared launch (kept off the stack)
thread_local SfxAngles g_angles;
thread_local dim3 g_fused_grid;
thread_local bool g_fused_ready = false;
thread_local bool g_fused_multi = false;      // the prepared launch runs the pairs in turn
}  // namespace

cudaError_t prepare_attn_fused(const AttnParams& a, const FusedSpec& f) {
    (void)cudaGetLastError();
    g_fused_ready = false;
    FusedTcParams& p = g_fused;
    g_fused_multi = f.pairs_in_turn != 0;
    cudaError_t e = g_fused_multi ? prepare_tc<true, true>(a, p.t, g_fused_grid)
                                  : prepare_tc<true, false>(a, p.t, g_fused_grid);
    if (e != cudaSuccess) return e;
    if (a.batch > kMaxFusedReq || a.layer0 != 0 || p.t.sq_pitch != a.sq || f.req_occ[0] != 0 ||
        f.req_occ[a.batch] > kMaxFusedOcc)
        return cudaErrorInvalidValue;
    const int64_t prow = (int64_t)a.lq * f.pool_slots;
    const int64_t crow = (int64_t)a.lq * a.rows;
    const int64_t srow = (int64_t)a.lq * a.batch_total * a.sq;
    if (prow > 0x7fffffffLL || crow > 0x7fffffffLL || srow > 0x7fffffffLL) return cudaErrorInvalidValue;
    if (!f.k_suf || !f.v_suf || !f.occ_cs || !f.sfx_cs) return cudaErrorInvalidValue;
    const cuuint64_t str[2] = {(cuuint64_t)HD * 2, (cuuint64_t)a.hkv * HD * 2};
    const cuuint32_t box128[3] = {64, 1, (cuuint32_t)BN};
    const cuuint32_t box64[3] = {64, 1, 64};
    const cuuint32_t box8[3] = {64, 1, 8};
    {   // pool [L*pool_slots][Hkv][128] in 128-, 64- and 8-row boxes: the pool stays put, so
        // the maps of the last call are reused while it is the same pool
        static thread_local const void* key_k = nullptr;
        static thread_local const void* key_v = nullptr;
        static thread_local int64_t key_rows = -1, key_hkv = -1;
        if (key_k != f.pool_k || key_v != f.pool_v || key_rows != prow || key_hkv != a.hkv) {
            key_k = nullptr;
            const cuuint64_t pdims[3] = {HD, (cuuint64_t)a.hkv, (cuuint64_t)prow};
            if (!encode(&p.tm_pk, f.pool_k, 3, pdims, str, box128) ||
                !encode(&p.tm_pv, f.pool_v, 3, pdims, str, box128) ||
                !encode(&p.tm_pk64, f.pool_k, 3, pdims, str, box64) ||
                !encode(&p.tm_pv64, f.pool_v, 3, pdims, str, box64) ||
                !encode(&p.tm_pk8, f.pool_k, 3, pdims, str, box8) ||
                !encode(&p.tm_pv8, f.pool_v, 3, pdims, str, box8))
                return cudaErrorInvalidValue;
            key_k = f.pool_k;
            key_v = f.pool_v;
            key_rows = prow;
            key_hkv = a.hkv;
        }
    }
    {   // suffix V [Lq*Btot*Sq][Hkv][128] in 128-, 64- and 8-row boxes
        const cuuint64_t sdims[3] = {HD, (cuuint64_t)a.hkv, (cuuint64_t)srow};
        if (!encode(&p.tm_sv, f.v_suf, 3, sdims, str, box128) ||
            !encode(&p.tm_sv64, f.v_suf, 3, sdims, str, box64) ||
            !encode(&p.tm_sv8, f.v_suf, 3, sdims, str, box8))
            return cudaErrorInvalidValue;
    }
    p.pool_k = f.pool_k;
    p.pool_v = f.pool_v;
    p.k_suf = f.k_suf;
    p.v_suf = f.v_suf;
    p.cache_k = const_cast<void*>(a.cache_k);
    p.cache_v = const_cast<void*>(a.cache_v);
    p.pos = f.pos;
    p.occ_cs = f.occ_cs;
    p.sfx_cs = f.sfx_cs;
    p.n_occ = f.req_occ[a.batch];
    g_angles.tab = f.sfx_cs;
    g_angles.sq = a.sq;
    g_angles.batch = a.batch;
    g_angles.rope = f.rope;
    std::memcpy(g_angles.req, a.req, sizeof(ReqParam) * (size_t)a.batch);
    p.pool_slots = f.pool_slots;
    p.rope = f.rope;
    std::memcpy(p.req_occ, f.req_occ, sizeof(int32_t) * (size_t)(a.batch + 1));
    std::memcpy(p.occ, f.occ, sizeof(FusedOcc) * (size_t)f.req_occ[a.batch]);
    g_fused_ready = true;
    return cudaSuccess;
}

cudaError_t launch_attn_fused(cudaStream_t s, Hook before) {
    if (!g_fused_ready) return cudaErrorInvalidValue;
    g_fused_ready = false;
    before();
    // the suffix angles on a few CTAs, then the fused kernel as its programmatic dependent
    const int64_t n = (int64_t)g_angles.batch * g_angles.sq * 64;
    const unsigned blocks = (unsigned)std::min<int64_t>(32, (n + 255) / 256);
    suffix_angles_kernel<<<blocks, 256, 0, s>>>(g_angles);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = g_fused_grid;
    cfg.blockDim = dim3(kThreadsFused);
    cfg.dynamicSmemBytes = kSmemBytes;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = g_fused_multi ? cudaLaunchKernelEx(&cfg, attn_tc_kernel<true, true>, g_fused)
                      : cudaLaunchKernelEx(&cfg, attn_tc_kernel<true, false>, g_fused);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

}  // namespace c2kv
