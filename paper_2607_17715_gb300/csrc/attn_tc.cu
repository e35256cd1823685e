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
#include <cuda.h>
#include <cudaTypedefs.h>

#include <math_constants.h>

#include <cstring>

#include "internal.cuh"
#include "ptx.cuh"

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
constexpr int NBAR = B_OD + 1;

constexpr int kSmemTiles = 2 /*Q_A, Q_B*/ + KSTAGES + VSTAGES;
constexpr size_t kSmemBytes = 1024 /*align*/ + (size_t)TILE * kSmemTiles + 8 * NBAR + 16;
static_assert(kSmemBytes <= 232448, "shared memory budget of one sm_100 CTA");

struct TcParams {                // CUtensorMap members carry their own alignment
    CUtensorMap tm_q;        // q_rot   [Lq*Btot][Sq'][Hq][128] box {64, G, TQ, 1}; Sq' = sq_pitch
    CUtensorMap tm_k;        // cache K [L*rows][Hkv][128]      box {64, 1, 128}
    CUtensorMap tm_v;        // cache V, same
    void* out;
    float* lse;
    int32_t* err;
    int64_t rows;
    int32_t layer0, lq, batch, batch_total, b0, sq, sq_pitch, hq, hkv, group, tq;
    float scale_log2;
    int32_t n_split;
    float* part_o;
    float* part_lse;
    ReqParam req[kMaxReq];
};

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

// ------------------------------------------------------------------ kernel

// One softmax thread's work on tile x (A or B) for every key tile, then its epilogue.
// r = TMEM lane (row within the tile), t0 = first suffix token of the tile.
__device__ __forceinline__ void softmax_tile(const TcParams& P, uint32_t tmem, uint32_t sBar, int x,
                                            int quad, int lane, int t0, int l, int bl, int b,
                                            int hk, int sp, int j_base, int n_kv,
                                            volatile uint32_t* abort) {
    auto bar = [&](int i) { return sBar + 8u * (uint32_t)i; };
    const int G = P.group;
    const int s_r = P.req[bl].n_slots;
    const int r = quad * 32 + lane;                 // row = TMEM lane
    const uint32_t lane_addr = (uint32_t)(quad * 32) << 16;
    const uint32_t colS = kColS + (uint32_t)x * BN;  // S_x, and P_x over its first 64 columns
    const uint32_t colO = kColO + (uint32_t)x * HD;
    const int t_row = min(t0 + r / G, P.sq - 1);    // rows past the suffix mirror its end
    const int lim = s_r + t_row;                    // last key this row may see
    const float sc = P.scale_log2;
    float m_run = -CUDART_INF_F;
    float l_run = 0.f;

    for (int j = 0; j < n_kv; ++j) {
        mbar_wait(bar(B_SF + x), (uint32_t)j & 1u, P.err, abort);
        tc_fence_after();
        uint32_t sv[4][32];
#pragma unroll
        for (int c = 0; c < 4; ++c) tmem_ld32(tmem + lane_addr + colS + c * 32, sv[c]);
        tmem_ld_wait();

        const int kbase = (j_base + j) * BN;
        if (kbase + BN - 1 > lim) {
#pragma unroll
            for (int c = 0; c < 4; ++c)
#pragma unroll
                for (int e = 0; e < 32; ++e)
                    if (kbase + c * 32 + e > lim) sv[c][e] = __float_as_uint(-CUDART_INF_F);
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

        // S_x(j) complete implies P_x(j-1).V(j-1) complete: O_x is current and may be scaled
        if (j >= 1 && __any_sync(0xffffffffu, resc)) {
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

    // ---------------------------------------------------------------- epilogue
    if (n_kv > 0) {
        mbar_wait(bar(B_OD), 0u, P.err, abort);
        tc_fence_after();
    }
    const int t = t0 + r / G;
    const int g = r - (r / G) * G;
    const bool any = l_run > 0.f;                 // some key of this split was visible
    const float inv = any ? 1.0f / l_run : 0.f;
    const int64_t row_id = (((int64_t)l * P.batch_total + b) * P.sq_pitch + t) * P.hq + hk * G + g;
    const int64_t lse_id = (((int64_t)l * P.batch_total + b) * P.hq + hk * G + g) * P.sq_pitch + t;
    if (P.n_split == 1) {
        __nv_bfloat16* orow = static_cast<__nv_bfloat16*>(P.out) + row_id * HD;
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            uint32_t ov[32];
            tmem_ld32(tmem + lane_addr + colO + c * 32, ov);
            tmem_ld_wait();
            if (t < P.sq) {
#pragma unroll
                for (int q8 = 0; q8 < 4; ++q8) {
                    uint4 w;
                    w.x = pack_bf16(__uint_as_float(ov[q8 * 8 + 0]) * inv, __uint_as_float(ov[q8 * 8 + 1]) * inv);
                    w.y = pack_bf16(__uint_as_float(ov[q8 * 8 + 2]) * inv, __uint_as_float(ov[q8 * 8 + 3]) * inv);
                    w.z = pack_bf16(__uint_as_float(ov[q8 * 8 + 4]) * inv, __uint_as_float(ov[q8 * 8 + 5]) * inv);
                    w.w = pack_bf16(__uint_as_float(ov[q8 * 8 + 6]) * inv, __uint_as_float(ov[q8 * 8 + 7]) * inv);
                    *reinterpret_cast<uint4*>(orow + c * 32 + q8 * 8) = w;
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
                for (int q4 = 0; q4 < 8; ++q4) {
                    float4 w = make_float4(__uint_as_float(ov[q4 * 4 + 0]) * inv, __uint_as_float(ov[q4 * 4 + 1]) * inv,
                                           __uint_as_float(ov[q4 * 4 + 2]) * inv, __uint_as_float(ov[q4 * 4 + 3]) * inv);
                    *reinterpret_cast<float4*>(orow + c * 32 + q4 * 4) = w;
                }
            }
        }
        if (t < P.sq)
            P.part_lse[(int64_t)sp * part_rows + lse_id] = any ? m_run + log2f(l_run) : -CUDART_INF_F;
    }
}

// The MMA issuer (one thread).  The tensor core's queue holds about one MMA, so anything
// the issuing thread does between two MMAs idles it, and a branch there costs about as much
// as an MMA.  So the descriptors are precomputed, the issue blocks are straight-line code,
// the kernel is specialised on whether the CTA has a tile B, and the ring stages and
// barrier parities advance by selects rather than branches.  Each block waits for its own
// inputs only: waiting for a later block's P inside an S block would hold that S back until
// the other tile's softmax finished, putting the two softmaxes in series.
template <bool kHasB>
__device__ __forceinline__ void mma_issuer(const TcParams& P, uint32_t tmem, uint32_t sQ, uint32_t sK,
                                           uint32_t sV, uint32_t sBar, int n_kv,
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
    // one key tile j >= 1:  PV_A(j-1)  S_A(j)  PV_B(j-1)  S_B(j)
    //   ks, kph: K stage and fill parity of tile j;  vs, vph: V stage and parity of tile j-1;
    //   pp: parity of P_x(j-1);  acc0: 0 only for the first P.V (j == 1)
    auto tile = [&](int ks, uint32_t kph, int vs, uint32_t vph, uint32_t pp, uint32_t acc0) {
        const uint64_t dk = dK0 + (uint64_t)ks * kTileDesc;
        const uint64_t dv = dV0 + (uint64_t)vs * kTileDesc;
        wait(B_PF + 0, pp);
        wait(B_VF + vs, vph);
        pv_block(tS_a, dv, tO_a, acc0);
        wait(B_KF + ks, kph);
        s_block(dQa, dk, tS_a);
        mma_commit(bar(B_SF + 0));
        if (kHasB) {
            wait(B_PF + 1, pp);
            pv_block(tS_b, dv, tO_b, acc0);
        }
        mma_commit(bar(B_VE + vs));
        if (kHasB) {
            s_block(dQb, dk, tS_b);
            mma_commit(bar(B_SF + 1));
        }
        mma_commit(bar(B_KE + ks));
    };

    wait(B_Q, 0u);
    wait(B_KF + 0, 0u);
    // key tile 0: S_A(0), S_B(0)
    s_block(dQa, dK0, tS_a);
    mma_commit(bar(B_SF + 0));
    if (kHasB) {
        s_block(dQb, dK0, tS_b);
        mma_commit(bar(B_SF + 1));
    }
    mma_commit(bar(B_KE + 0));
    // tiles 1 .. n_kv-1, ring positions advanced without branches
    int ks = 1, vs = 0;
    uint32_t kph = 0u, vph = 0u, acc0 = 0u;
    for (int j = 1; j < n_kv; ++j) {
        tile(ks, kph, vs, vph, (uint32_t)(j - 1) & 1u, acc0);
        acc0 = 1u;
        const bool kw = ks == KSTAGES - 1;
        ks = kw ? 0 : ks + 1;
        kph ^= kw ? 1u : 0u;
        const bool vw = vs == VSTAGES - 1;
        vs = vw ? 0 : vs + 1;
        vph ^= vw ? 1u : 0u;
    }
    // last P.V pair: P_x(n_kv - 1), V stage (n_kv - 1) % 2
    const int vl = vs;
    const uint32_t vphl = vph;
    const uint32_t pl = (uint32_t)(n_kv - 1) & 1u;
    const uint64_t dvl = dV0 + (uint64_t)vl * kTileDesc;
    wait(B_PF + 0, pl);
    wait(B_VF + vl, vphl);
    pv_block(tS_a, dvl, tO_a, acc0);
    if (kHasB) {
        wait(B_PF + 1, pl);
        pv_block(tS_b, dvl, tO_b, acc0);
    }
    mma_commit(bar(B_VE + vl));
    mma_commit(bar(B_OD));
}

__global__ void __launch_bounds__(kThreads, 1) attn_tc_kernel(const __grid_constant__ TcParams P) {
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
    const int s_r = P.req[bl].n_slots;
    // pair of Q tiles, the last first: under a causal mask the later pairs see more keys, so
    // the longest CTAs start in the first wave
    const int pr = (int)(gridDim.x / P.n_split) - 1 - (int)(blockIdx.x / P.n_split);
    const int sp = (int)(blockIdx.x % P.n_split);   // key-range split
    const int t0a = 2 * pr * P.tq;
    const int t0b = t0a + P.tq;
    const bool has_b = t0b < P.sq;
    const int t_last = min(P.sq - 1, (has_b ? t0b : t0a) + P.tq - 1);
    const int n_kv_all = (s_r + t_last + 1 + BN - 1) / BN;
    // this CTA's key tiles: [j_base, j_base + n_kv) of the request's n_kv_all
    const int per_split = (n_kv_all + P.n_split - 1) / P.n_split;
    const int j_base = sp * per_split;
    const int n_kv = max(0, min(n_kv_all, j_base + per_split) - j_base);

    if (threadIdx.x == 0) {
        mbar_init(bar(B_Q), 1);
        for (int s = 0; s < KSTAGES; ++s) {
            mbar_init(bar(B_KF + s), 1);
            mbar_init(bar(B_KE + s), 1);
        }
        for (int s = 0; s < VSTAGES; ++s) {
            mbar_init(bar(B_VF + s), 1);
            mbar_init(bar(B_VE + s), 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(bar(B_SF + i), 1);
            mbar_init(bar(B_PF + i), 128);
        }
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

    if (warp < 4) {
        asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(kRegsLow));
        if (warp == 0 && lane == 0 && n_kv > 0) {
            // ------------------------------------------------------------ TMA producer
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&P.tm_q)) : "memory");
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&P.tm_k)) : "memory");
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&P.tm_v)) : "memory");
            const int qz = l * P.batch_total + b;
            mbar_expect_tx(bar(B_Q), has_b ? 2 * TILE : TILE);
            tma_load_4d(sQ, &P.tm_q, 0, hk * G, t0a, qz, bar(B_Q));
            tma_load_4d(sQ + HALF_TILE, &P.tm_q, 64, hk * G, t0a, qz, bar(B_Q));
            if (has_b) {
                tma_load_4d(sQ + TILE, &P.tm_q, 0, hk * G, t0b, qz, bar(B_Q));
                tma_load_4d(sQ + TILE + HALF_TILE, &P.tm_q, 64, hk * G, t0b, qz, bar(B_Q));
            }
            const int key0 = (int)((int64_t)(P.layer0 + l) * P.rows + P.req[bl].row_base) + j_base * BN;
            // two independent queues: a K load waits only for its own K stage
            int jk = 0, jv = 0;
            while (jk < n_kv || jv < n_kv) {
                if (jk < n_kv && (jk < KSTAGES || mbar_try(bar(B_KE + jk % KSTAGES),
                                                          (uint32_t)((jk / KSTAGES) - 1) & 1u))) {
                    const int s = jk % KSTAGES;
                    const int krow = key0 + jk * BN;
                    mbar_expect_tx(bar(B_KF + s), TILE);
                    tma_load_3d(sK + s * TILE, &P.tm_k, 0, hk, krow, bar(B_KF + s));
                    tma_load_3d(sK + s * TILE + HALF_TILE, &P.tm_k, 64, hk, krow, bar(B_KF + s));
                    ++jk;
                    continue;
                }
                if (jv < n_kv && (jv < VSTAGES || mbar_try(bar(B_VE + jv % VSTAGES),
                                                          (uint32_t)((jv / VSTAGES) - 1) & 1u))) {
                    const int s = jv % VSTAGES;
                    const int vrow = key0 + jv * BN;
                    mbar_expect_tx(bar(B_VF + s), TILE);
                    tma_load_3d(sV + s * TILE, &P.tm_v, 0, hk, vrow, bar(B_VF + s));
                    tma_load_3d(sV + s * TILE + HALF_TILE, &P.tm_v, 64, hk, vrow, bar(B_VF + s));
                    ++jv;
                    continue;
                }
                // nothing issuable: wait (bounded) for the stage the next K load needs
                if (jk < n_kv)
                    mbar_wait(bar(B_KE + jk % KSTAGES), (uint32_t)((jk / KSTAGES) - 1) & 1u, P.err, abort);
                else
                    mbar_wait(bar(B_VE + jv % VSTAGES), (uint32_t)((jv / VSTAGES) - 1) & 1u, P.err, abort);
            }
        } else if (warp == 1 && lane == 0 && n_kv > 0) {
            // ------------------------------------------------------------ MMA issuer
            if (has_b)
                mma_issuer<true>(P, tmem, sQ, sK, sV, sBar, n_kv, abort);
            else
                mma_issuer<false>(P, tmem, sQ, sK, sV, sBar, n_kv, abort);
        }
    } else {
        asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(kRegsHigh));
        // ---------------------------------------------------------------- softmax warps
        const int x = warp >= 8 ? 1 : 0;               // tile A (warps 4..7) or B (8..11)
        if (x == 0 || has_b)
            softmax_tile(P, tmem, sBar, x, warp & 3, lane, x ? t0b : t0a, l, bl, b, hk, sp, j_base,
                         n_kv, abort);
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

// Merge the splits: lse = log2 sum_s 2^lse_s, O = sum_s 2^(lse_s - lse) O_s.  One warp per
// (layer, request, suffix token, query head) row; lane i owns head channels 4i .. 4i+3.
// Every split's lse and O slice is loaded before any is used (at most kMaxSplit), so the
// loads of one row are all in flight together.
constexpr int kMaxSplit = 16;

__global__ void __launch_bounds__(256) attn_combine_kernel(const __grid_constant__ AttnParams P) {
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
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    if (!fn) {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q{};
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    }
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
    attn_combine_kernel<<<(unsigned)blocks, 256, 0, s>>>(a);
    return cudaGetLastError();
}

bool attn_tc_supported(int dtype, int d, int hq, int hkv) {
    if (dtype != kDtypeBf16 || d != HD || hkv < 1 || hq % hkv) return false;
    const int g = hq / hkv;
    return g == 1 || g == 2 || g == 4 || g == 8 || g == 16;
}

cudaError_t launch_attn_tc(const AttnParams& a, cudaStream_t s, Hook before) {
    (void)cudaGetLastError();   // report this launch's error only, not a stale one
    cudaError_t e = cudaSuccess;
    static bool smem_set = false;           // once per process (one device per context)
    if (!smem_set) {
        e = cudaFuncSetAttribute(attn_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)kSmemBytes);
        if (e != cudaSuccess) return e;
        smem_set = true;
    }
    {   // the register split must not ask for more than the launch holds
        static int launch_regs = -1;
        if (launch_regs < 0) {
            cudaFuncAttributes fa{};
            e = cudaFuncGetAttributes(&fa, attn_tc_kernel);
            if (e != cudaSuccess) return e;
            launch_regs = fa.numRegs;
        }
        if (launch_regs * kThreads < 128 * kRegsLow + 256 * kRegsHigh) return cudaErrorInvalidConfiguration;
    }
    const int pitch = a.sq_pitch > 0 ? a.sq_pitch : a.sq;
    if (pitch < a.sq || (pitch != a.sq && a.n_split > 1)) return cudaErrorInvalidValue;
    TcParams p;
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
    std::memcpy(p.req, a.req, sizeof(ReqParam) * (size_t)a.batch);
    const int64_t pairs = ((a.sq + tq - 1) / tq + 1) / 2;
    const int64_t gx = pairs * p.n_split;
    if (gx > 0x7fffffffLL) return cudaErrorInvalidValue;
    const dim3 grid((unsigned)gx, a.hkv, a.lq * a.batch);
    if (grid.z > 65535u || grid.y > 65535u) return cudaErrorInvalidValue;
    before();
    attn_tc_kernel<<<grid, kThreads, kSmemBytes, s>>>(p);
    return cudaGetLastError();
}

}  // namespace c2kv
