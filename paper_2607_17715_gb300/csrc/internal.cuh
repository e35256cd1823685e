// Internal declarations shared by the C2KV library's translation units (not installed).
//
// Per-call metadata (chunk occurrences, per-request row layout, RoPE frequencies) travels
// inside the kernel parameter block, so compose and attend need no host-to-device copy
// and no device-side metadata buffer.
#pragma once

#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

namespace c2kv {

constexpr int kDtypeBf16 = 0;
constexpr int kDtypeF32 = 1;
constexpr int kMaxHalf = 64;        // head_dim / 2 for head_dim <= 128
constexpr int kMaxOcc = 512;        // chunk occurrences per compose launch (24 KB of parameters)
constexpr int kMaxReq = 256;        // requests per suffix / attention launch
constexpr int kMaxMergeSplits = 32; // key-range splits the tensor-core kernel merges itself
constexpr int kComposeTile = 16;    // most composed slots per compose tile (per layer)
constexpr int kComposeBulkTile = 32;   // most slots per tile of the bulk-copy compose kernel

// RoPE frequency i as a fraction of a full turn in 0.64 fixed point:
// turn[i] = round(theta^(-2i/d) / (2 pi) * 2^64).  For an integer position p the angle in
// turns is the low 64 bits of p * turn[i] (a phase accumulator: wrap-around is the
// reduction modulo 2 pi, exact in integers), so no large float angle is ever formed.
struct RopeTurns {
    uint64_t turn[kMaxHalf];
};

// One chunk occurrence of a compose launch.
struct OccParam {
    int32_t src_base;    // first pool slot of the chunk (pool chunks)
    int32_t dest_row;    // first composed row
    int32_t delta;       // positions to turn by (o_i, or 0 under fixed_pos)
    int32_t n;           // original chunk length
    int32_t k;           // ratio
    int32_t m;           // slots
    int32_t tile_base;   // first compose tile of this occurrence (prefix over the launch)
    int32_t host;        // 1: the chunk stays in host memory, read through host_k / host_v
    const void* host_k;  // device-accessible [L][m][Hkv][d] (host-resident chunks)
    const void* host_v;
};

// Everything of a compose launch but its occurrence table.
struct ComposeHead {
    const void* pool_k;      // [L][pool_slots][Hkv][d]
    const void* pool_v;
    void* out_k;             // [L][rows][Hkv][d]
    void* out_v;
    int32_t* pos;            // [rows]
    int32_t* err;            // device error word: bit 0 = index refused
    int64_t pool_slots;
    int64_t rows;
    int32_t n_occ;
    int32_t n_tiles;
    int32_t hkv;
    int32_t layer0;          // layer of grid row 0 (a launch covers layers layer0 .. + gridDim.y)
    int32_t tile_slots;      // composed slots per tile, 1 .. kComposeTile (1 .. kComposeBulkTile
                             // with bulk; chosen per launch)
    int32_t bulk;            // 1: the bulk-copy kernel (every chunk in the device pool)
    int32_t pre_rope;        // 1: stored K is before RoPE; slot j of occurrence o turns by its
                             // composed position o.delta + p_j (PRE_ROPE storage)
    RopeTurns rope;
};

struct ComposeParams : ComposeHead {
    OccParam occ[kMaxOcc];
};

struct CompressParams {
    const void* in_k;        // [L][rows_in][Hkv][d]
    const void* in_v;
    void* pool_k;            // [L][pool_slots][Hkv][d]
    void* pool_v;
    int64_t pool_slots;
    int32_t slot_base;
    int32_t m;               // slots
    int32_t n;               // tokens
    int32_t k;               // ratio
    int32_t rows_in;         // n (meanpool) or m (provided)
    int32_t one_row;         // 1 = provided (slot j is input row j); 0 = block mean
    int32_t layers;
    int32_t hkv;
    int32_t turn;            // 1: K turned to the slot's local position p_j (LOCAL_ROPE
                             // storage); 0: kept before RoPE (PRE_ROPE)
    RopeTurns rope;
};

struct ReqParam {
    int32_t row_base;        // first cache row of the request
    int32_t n_slots;         // composed slots S_r
    int32_t l_req;           // composed span L_r (suffix token t sits at L_r + t)
    int32_t t0;              // suffix index of this launch's first token (0 for attend; the
                             // decode step for decode)
};

struct SuffixParams {
    const void* q;           // [Lq][B][Sq][Hq][d]   (B = this launch's requests)
    const void* k;           // [Lq][B][Sq][Hkv][d]
    const void* v;
    void* q_rot;             // [Lq][B][Sq][Hq][d]
    void* cache_k;           // [L][rows][Hkv][d]
    void* cache_v;
    int32_t* pos;            // [rows]
    int64_t rows;
    int32_t layer0;          // first cache layer touched
    int32_t lq;              // layers in this call
    int32_t batch;           // requests in this launch
    int32_t batch_total;     // requests in the q / out tensors
    int32_t b0;              // first request of this launch
    int32_t sq;
    int32_t hq;
    int32_t hkv;
    int32_t pad_rows;        // 1: zero each request's rows from pad_from up to the next 128-row
                             // boundary
    RopeTurns rope;
    ReqParam req[kMaxReq];
    int32_t pad_from[kMaxReq];   // request-relative row where the zeroing starts (the row after
                                 // the suffix; at a 128-row boundary for none)
};

struct AttnParams {
    const void* q_rot;       // [Lq][Btot][Sq'][Hq][d], Sq' = sq_pitch
    const void* cache_k;     // [L][rows][Hkv][d]
    const void* cache_v;
    void* out;               // [Lq][Btot][Sq'][Hq][d]
    float* lse;              // [Lq][Btot][Hq][Sq'] or null
    int32_t* err;            // device error word: bit 1 = a bounded wait expired
    int64_t rows;
    int32_t layer0;
    int32_t lq;
    int32_t batch;
    int32_t batch_total;
    int32_t b0;
    int32_t sq;
    int32_t sq_pitch;        // tokens allocated per (layer, request) in q_rot, out and lse:
                             // rows sq .. sq_pitch-1 are neither read nor written; 0 = sq
                             // (tensor-core kernel only, and only with n_split == 1)
    int32_t hq;
    int32_t hkv;
    float scale_log2;        // log2(e) / sqrt(d)
    int32_t n_split;         // key-range splits per work unit (1 = write O directly)
    float* part_o;           // n_split > 1: [n_split][Lq][Btot][Sq][Hq][d] fp32, normalised
    float* part_lse;         // n_split > 1: [n_split][Lq][Btot][Hq][Sq] fp32, log2 domain
    int32_t pairs_per_cta;   // tensor-core kernel: at most this many pairs of query tiles per
                             // CTA (0 = chosen per launch)
    int32_t dependent;       // tensor-core kernel and its merge: launched as the programmatic
                             // dependent of the kernel before them on the stream (each waits
                             // for that grid before it reads memory)
    uint32_t* tickets;       // tensor-core kernel with n_split > 1: null (attn_combine_kernel
                             // merges), or one zeroed counter per (layer, request, KV head,
                             // pair): the unit's last split merges the partials in the kernel
                             // and sets it back to zero
    int32_t key_pingpong;    // tensor-core kernel: a pair with one query tile (a decode step's)
                             // splits its key tiles between the two softmax warpgroups, merged
                             // at the end (a different rounding order: off where the result must
                             // equal the fused kernel's bit for bit)
    int32_t sif_k;           // tensor-core kernel, extraction C2 rows (Sec. 3.3.1): 0, or the
                             // ratio k: the request's n_slots key rows are then the chunk's n
                             // document tokens, suffix token j is C2 token c_j, and of the
                             // document keys row j sees only the sink block [0, min(k, n)) and
                             // its own block [jk, min((j+1)k, n)); n_split must be 1
    ReqParam req[kMaxReq];
};

// Called by a launcher after its host-side preparation (tensor maps, function attributes)
// and right before it enqueues its kernels, so that a trace event recorded there brackets
// device work only.
struct Hook {
    void (*fn)(void*) = nullptr;
    void* arg = nullptr;
    void operator()() const {
        if (fn) fn(arg);
    }
};

// Launchers: return the launch error, never throw.  `d` is head_dim.
// max_ctas > 0 caps the CTAs per layer; each then walks several tiles (a compose that reads
// host-resident chunks is bound by the host link, and leaves the other SMs to attention).
cudaError_t launch_compose(const ComposeParams& p, int dtype, int d, int layers, cudaStream_t s,
                           int max_ctas = 0, Hook pre = {});
cudaError_t launch_compress(const CompressParams& p, int dtype, int d, cudaStream_t s);
cudaError_t launch_suffix_prep(const SuffixParams& p, int dtype, int d, cudaStream_t s);
cudaError_t launch_attn_simt(const AttnParams& p, int dtype, int d, cudaStream_t s);


// Decode attention (decode.cu): one new token per request (suffix index ReqParam::t0,
// already rotated into q_rot and appended to the cache) over keys 0 .. S_r + t0.
struct DecodeParams {
    const void* q_rot;       // [Lq][Btot][Hq][d]
    const void* cache_k;     // [L][rows][Hkv][d]
    const void* cache_v;
    void* out;               // [Lq][Btot][Hq][d]
    float* lse;              // [Lq][Btot][Hq] or null
    float* part_o;           // n_split > 1: [n_split][Lq][Btot][Hq][d] fp32, normalised
    float* part_lse;         // n_split > 1: [n_split][Lq][Btot][Hq] fp32, log2 domain
    int32_t* err;            // device error word: bit 1 = a bounded wait expired
    int64_t rows;
    int32_t layer0;
    int32_t lq;
    int32_t batch;
    int32_t batch_total;
    int32_t b0;
    int32_t hq;
    int32_t hkv;
    int32_t d;
    int32_t n_split;         // key-range splits per (layer, request, KV head)
    int32_t keys_per_split;
    float scale_log2;        // log2(e) / sqrt(d)
    int32_t dependent;       // launched as the programmatic dependent of the suffix kernel that
                             // writes this step's query and key row (nothing between them)
    ReqParam req[kMaxReq];
};
bool decode_supported(int dtype, int d, int hq, int hkv);
cudaError_t launch_decode(const DecodeParams& p, int dtype, cudaStream_t s, Hook before = {});

// SIF-masked extraction attention (extract.cu): one attention layer of the extractor over
// a chunk's n document tokens and m = ceil(n/k) C2 tokens, [x_0..x_{n-1}; c_0..c_{m-1}].
struct ExtractParams {
    const void* q;           // [Lq][n_all][Hq][d] pre-RoPE
    const void* k;           // [Lq][n_all][Hkv][d] pre-RoPE
    const void* v;           // [Lq][n_all][Hkv][d]
    void* q_rot;             // scratch, shaped like q
    void* k_rot;             // scratch, shaped like k
    void* out;               // [Lq][n_all][Hq][d]
    float* lse;              // [Lq][Hq][n_all] or null
    int32_t* err;            // device error word (bounded waits of the tensor-core kernel)
    int32_t lq;
    int32_t n;               // document tokens
    int32_t ratio;           // k, the block size
    int32_t n_all;           // n + ceil(n / k)
    int32_t hq;
    int32_t hkv;
    float scale_log2;
    int32_t pairs_per_cta;   // the tensor-core attention launches' AttnParams::pairs_per_cta
    RopeTurns rope;
};
// With s2 (and the events fork and join), the tensor-core route runs the C2 rows' attention on
// s2, beside the document rows' attention on s; the work ends on s.
cudaError_t launch_extract(const ExtractParams& p, int dtype, int d, cudaStream_t s,
                           cudaStream_t s2 = nullptr, cudaEvent_t fork = nullptr, cudaEvent_t join = nullptr);
// Whether launch_extract takes the tensor-core route; otherwise every row runs on the CUDA
// cores.
bool extract_uses_tc(int dtype, int d, int hq, int hkv);

// Tiled tensor map for TMA (cuTensorMapEncodeTiled through the runtime's driver entry point);
// false when the driver refuses it (attn_tc.cu).
bool encode_tensor_map(CUtensorMap* tm, CUtensorMapDataType type, int rank, const void* base,
                       const cuuint64_t* dims, const cuuint64_t* strides_bytes, const cuuint32_t* box,
                       CUtensorMapSwizzle swizzle);

// Tensor-core attention (attn_tc.cu).
bool attn_tc_supported(int dtype, int d, int hq, int hkv);
cudaError_t launch_attn_tc(const AttnParams& p, cudaStream_t s, Hook before = {});
// Merge n_split partial (O, lse) over disjoint key ranges into out (bf16) and lse (attn_tc.cu).
cudaError_t launch_attn_combine(const AttnParams& p, cudaStream_t s);
// CTAs of one tensor-core attention launch before key-range splitting.
int64_t attn_tc_units(int hq, int hkv, int sq, int lq, int batch);

// Fused compose + attention (attn_tc.cu): the attention reads the composed slots straight
// from the chunk pool, turns K by its occurrence's offset in shared memory, and writes the
// composed cache (K', V, positions) as it goes.  The suffix rows must already be in the
// cache (suffix preparation first).
struct FusedOcc {
    int32_t src_row;         // first pool slot of the chunk
    int32_t dest_row;        // first composed row, relative to the request's row_base
    int32_t m;               // slots
    int32_t delta;           // positions to turn by
    int32_t n;               // original chunk length
    int32_t k;               // ratio
};
// The fused launch carries its occurrence table and per-request ranges in its parameter block,
// and a launch's latency grows with that block (about 0.4 us per KB on a GB300: the 32-layer
// fused step took 92.7 us with room for 512 occurrences and 256 requests, 88.1 us with 32
// occurrences).  So the fused route takes at most 128 occurrences of at most 32 requests;
// larger calls compose, then attend.
constexpr int kMaxFusedOcc = 128;
constexpr int kMaxFusedReq = 32;
struct FusedSpec {
    const void* pool_k;      // [L][pool_slots][Hkv][128]
    const void* pool_v;
    const void* k_suf;       // [L][B][Sq][Hkv][128]: the suffix rows before RoPE (K) and V
    const void* v_suf;
    int32_t* pos;            // [rows]
    float2* occ_cs;          // scratch [L][occurrences][64]: (cos, sin) of each occurrence's
                             // turn, filled by the kernel
    float2* sfx_cs;          // scratch [B][Sq][64]: (cos, sin) of each suffix token's position,
                             // filled by a small kernel launched just before
    int32_t pairs_in_turn;   // 1: a CTA runs every pair of query tiles of its (layer, request,
                             // KV head), the last pair first, which composes the cache
    int64_t pool_slots;
    RopeTurns rope;
    int32_t req_occ[kMaxFusedReq + 1];   // request i of the launch: occurrences [req_occ[i], req_occ[i+1])
    FusedOcc occ[kMaxFusedOcc];
};
// Host preparation (tensor maps, parameters) of a fused launch, then the launch.  The fused
// kernel also does the suffix preparation (the queries and the suffix keys turned in shared
// memory, the suffix rows and the zero rows up to the next 128-row boundary written to the
// cache): the AttnParams' q_rot is the queries before RoPE.
cudaError_t prepare_attn_fused(const AttnParams& a, const FusedSpec& f);
cudaError_t launch_attn_fused(cudaStream_t s, Hook before = {});

// Loads (under CUDA's lazy module loading) the kernels of a translation unit that
// c2kv_attend_noalloc can launch for this dtype and head_dim, so that launching them later
// takes no device memory.
cudaError_t preload_suffix_kernels(int dtype, int d);      // kv_kernels.cu
cudaError_t preload_attn_simt_kernels(int dtype, int d);   // attn_simt.cu
cudaError_t preload_attn_tc_kernels();                     // attn_tc.cu
// The device address of c2kv_attend_noalloc's fixed scratch array on the current device, its
// module loaded, with every kernel that call can launch (noalloc.cu); called by c2kv_create.
cudaError_t noalloc_prepare(int dtype, int d, bool tc, void** scratch);

// Where a caller's tensor lives: device (or managed) memory, pinned host memory the GPU can
// address (mapped, same address on both sides), or memory the CUDA runtime does not know
// (which no kernel may dereference).  NULL counts as device memory.
enum class MemKind { kDevice, kHost, kUnknown };
MemKind mem_kind(const void* p);

// Read-only view of a context and one of its caches, for entry points defined outside
// c2kv_api.cu (c2kv_attend_noalloc).
struct AttendView {
    int32_t layers, n_q_heads, n_kv_heads, head_dim, dtype, attn_impl, attn_pairs;
    int device;              // the context's device
    void* noalloc_scratch;   // c2kv_attend_noalloc's fixed array on that device
    cudaStream_t stream;
    int32_t* err;
    RopeTurns turns;
    void* cache_k;
    void* cache_v;
    int32_t* pos;
    int64_t rows;
    int32_t batch;
    int32_t suffix_capacity;
    const int32_t* row_base;
    const int32_t* n_slots;
    const int32_t* l_req;
};

}  // namespace c2kv

struct c2kv_ctx;
struct c2kv_cache;
namespace c2kv {
// Fills `v` if `cache` belongs to `ctx` (returns false otherwise).
bool attend_view(const c2kv_ctx* ctx, const c2kv_cache* cache, AttendView* v);
// Records that a suffix of n_suffix tokens over layers [l0, l0 + n) was written, with the
// rows after it zeroed up to the 128-row edge (what a later decode step reads as finite).
void note_suffix_written(c2kv_cache* cache, int32_t l0, int32_t n, int32_t n_suffix);
// Records `msg` as the context's last error and returns `code`.
int32_t set_last_error(c2kv_ctx* ctx, int32_t code, const char* msg);
}  // namespace c2kv
