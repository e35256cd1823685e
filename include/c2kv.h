/*
 * c2kv.h -- C ABI of the GB300 (sm_103a) library for C2KV compressed, composable KV-cache
 * reuse (arXiv 2607.17715): store per-chunk compressed KV, compose the chunks a request
 * asks for into one contiguous GQA cache (RoPE re-rotated to the request's positions),
 * and run the request's suffix tokens' attention over it.
 *
 * The paper's generalized reuse pipeline (Sec. 2.2) has three steps, and the calls below
 * follow them:
 *   Encoding  M : KV_k     = M(x_k)                   -> c2kv_compress_chunk
 *   Blending  B : KV_total = B(x_s, KV_1 .. KV_K)     -> c2kv_compose
 *   Inference F : y        = F([KV_total, x_q])       -> c2kv_attend
 *
 * Conventions shared by every call
 *   - Every call returns a c2kv_status at once: C2KV_OK (0) or a negative code.  No C++
 *     exception and no abort ever crosses this boundary.
 *   - GPU work is enqueued on the context's CUDA stream and runs asynchronously.  Errors
 *     found by a kernel's own bounds checks surface at the next c2kv_sync().
 *   - On any error status the library's state (pool, chunk table, caches) is unchanged
 *     and c2kv_last_error() describes the failure.
 *   - Tensors are dense, row-major, with the innermost dimension last.  "d" is head_dim,
 *     "Hq"/"Hkv" the query / key-value head counts, "L" the layer count.  Element type is
 *     the context dtype (bf16 or fp32) unless stated.
 *   - The caller owns every buffer it passes in; the library owns the chunk pool and the
 *     composed caches it returns.
 *   - Tensor pointers passed in must be 16-byte aligned (fp32 lse arrays: 4-byte), since
 *     the kernels move rows in 16-byte vectors and by TMA; others give ERR_ARG.
 *   - A context is used from one host thread at a time.
 */
#ifndef C2KV_H
#define C2KV_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef int32_t c2kv_status;

#define C2KV_OK                  0
#define C2KV_ERR_ARG            -1   /* null pointer, bad size or shape                  */
#define C2KV_ERR_DTYPE          -2   /* dtype not supported for this call                */
#define C2KV_ERR_NOMEM          -3   /* device or pinned host allocation failed          */
#define C2KV_ERR_POOL_FULL      -4   /* no contiguous free slot range in the chunk pool  */
#define C2KV_ERR_BAD_CHUNK      -5   /* unknown or freed chunk id                        */
#define C2KV_ERR_POSITIONS      -6   /* offsets negative, decreasing or overlapping      */
#define C2KV_ERR_CUDA           -7   /* a CUDA runtime call failed                       */
#define C2KV_ERR_DEVICE_BOUNDS  -8   /* a kernel's bounds check refused an index         */
#define C2KV_ERR_STATE          -9   /* object used in the wrong state / wrong context   */
#define C2KV_ERR_UNSUPPORTED   -10   /* valid request this build does not implement      */

#define C2KV_DTYPE_BF16 0
#define C2KV_DTYPE_F32  1

/* c2kv_compress_chunk modes */
#define C2KV_MODE_MEANPOOL 0  /* tokens -> slots: block mean of pre-RoPE K/V rows            */
#define C2KV_MODE_PROVIDED 1  /* slots given pre-RoPE by an external extractor               */
#define C2KV_MODE_STORED   2  /* slots given already in stored form (load from host storage) */
#define C2KV_MODE_HOST     3  /* stored-form slots that stay in pinned host memory (no copy)   */

/* c2kv_attend kernel choice */
#define C2KV_ATTN_AUTO   0    /* tensor-core kernel where it applies, SIMT otherwise */
#define C2KV_ATTN_SIMT   1    /* CUDA-core fp32-accumulate kernel (any dtype)        */
#define C2KV_ATTN_TC     2    /* tcgen05 / TMEM tensor-core kernel (bf16, d = 128)    */

/* c2kv_config.storage: the form stored chunk K takes in the pool */
#define C2KV_STORAGE_LOCAL_ROPE 0   /* K carries RoPE at its chunk-local slot position p_j;
                                       compose turns it by the occurrence offset o_i      */
#define C2KV_STORAGE_PRE_ROPE   1   /* K kept before any positional embedding, as Sec. 3.3.1
                                       stores it; compose applies RoPE at o_i + p_j once   */

/* c2kv_compose_attend: when the fused compose + attention kernel runs */
#define C2KV_FUSE_AUTO   0    /* when each (layer, request, KV head) has a single pair of
                                 128-row query tiles, n_suffix * Hq / Hkv <= 256: every
                                 stored slot is then read and turned by exactly one CTA   */
#define C2KV_FUSE_NEVER  1    /* always compose, then attend                           */
#define C2KV_FUSE_ALWAYS 2    /* whenever the fused kernel takes the call; with several
                                 pairs of query tiles one CTA runs them in turn, the last
                                 pair composing the cache and the others reading it      */

typedef struct c2kv_ctx c2kv_ctx;
typedef struct c2kv_cache c2kv_cache;

/* Model / pool shape.  head_dim must be 64 or 128; n_q_heads a multiple of n_kv_heads. */
typedef struct c2kv_config {
    int32_t layers;
    int32_t n_q_heads;
    int32_t n_kv_heads;
    int32_t head_dim;
    double  rope_theta;        /* RoPE base: pair (i, i + d/2) turns by pos * theta^(-2i/d) */
    int32_t dtype;             /* C2KV_DTYPE_BF16 or C2KV_DTYPE_F32                           */
    int32_t pool_slots;        /* capacity of the device chunk pool, in slots (all layers)    */
    int32_t fixed_pos;         /* 1 = no re-rotation at compose ("Fixed-Pos." ablation,
                                  Sec. 4.8): slots keep their chunk-local positions          */
    int32_t attn_impl;         /* C2KV_ATTN_AUTO / _SIMT / _TC                                */
    int32_t attn_split;        /* tensor-core attention key-range splits per work unit:
                                  0 = chosen per call (split only when the units would leave
                                  most SMs idle), 1 = never, n <= 16 = always n (partials
                                  merged by an exact log-sum-exp combine)                     */
    int32_t fuse;              /* C2KV_FUSE_AUTO / _NEVER / _ALWAYS (c2kv_compose_attend)     */
    int32_t storage;           /* C2KV_STORAGE_LOCAL_ROPE (0) or C2KV_STORAGE_PRE_ROPE          */
    int32_t attn_pairs;        /* pairs of 128-row query tiles one tensor-core attention CTA
                                  runs in turn: 0 = chosen per launch (several only when the
                                  launch is many waves of CTAs), n >= 1 = n (fewer where a
                                  (layer, request, KV head) has fewer pairs)                  */
} c2kv_config;

/* Chunk metadata (c2kv_chunk_info). */
typedef struct c2kv_chunk_desc {
    int32_t n_tokens;          /* original chunk length n (the span it occupies when composed) */
    int32_t ratio_k;           /* compression ratio k                                          */
    int32_t n_slots;           /* m = ceil(n / k)                                              */
    int32_t slot_base;         /* first pool slot                                              */
    void*   k;                 /* device: pool K at (layer 0, slot_base); layer stride below   */
    void*   v;                 /* device: pool V, same layout                                  */
    int64_t layer_stride;      /* elements between layers = pool_slots * Hkv * d              */
} c2kv_chunk_desc;

/* Composed cache metadata (c2kv_cache_info).  Host arrays stay valid until release. */
typedef struct c2kv_cache_desc {
    int32_t batch;
    int32_t layers;
    int64_t rows;              /* rows per layer in k / v (all requests, padded)          */
    void*   k;                 /* device [layers][rows][Hkv][d]                            */
    void*   v;                 /* device [layers][rows][Hkv][d]                            */
    int32_t* pos;              /* device [rows]: composed position of each row             */
    const int32_t* row_base;   /* host [batch]: first row of each request (multiple of 128)*/
    const int32_t* n_slots;    /* host [batch]: composed slots S_r of each request         */
    const int32_t* l_req;      /* host [batch]: composed span L_r = max_i (o_i + n_i)      */
    const int32_t* capacity;   /* host [batch]: rows reserved for the request              */
    int32_t suffix_capacity;   /* suffix rows reserved after the slots of each request     */
} c2kv_cache_desc;

/* ABI version of this header (bumped on any incompatible change). */
#define C2KV_ABI_VERSION 5
int32_t c2kv_abi_version(void);

/*
 * c2kv_create -- make a context on the current CUDA device.
 *   cfg     : shape and pool size (copied).
 *   stream  : cudaStream_t to enqueue all work on (NULL = legacy default stream).
 *   out     : receives the context.
 * Allocates the chunk pool: 2 * layers * pool_slots * Hkv * d elements of device memory.
 * Errors: ERR_ARG (bad shape / null out), ERR_DTYPE, ERR_NOMEM, ERR_CUDA.
 */
c2kv_status c2kv_create(const c2kv_config* cfg, void* stream, c2kv_ctx** out);

/* c2kv_destroy -- synchronize the stream and free everything the context owns, including
 * composed caches not yet released.  NULL is accepted. */
c2kv_status c2kv_destroy(c2kv_ctx* ctx);

/* c2kv_set_stream -- switch the stream later calls enqueue on (e.g. torch's current one). */
c2kv_status c2kv_set_stream(c2kv_ctx* ctx, void* stream);

/*
 * c2kv_compress_chunk -- the encoding step M: store one chunk (document) as compressed
 * slots in the device pool.  Sec. 3.2.1: a chunk of n tokens gets m = ceil(n/k) slots, one
 * per block of k consecutive tokens; Sec. 3.3.1: slot j takes the position of the last
 * token of its block, p_j = min((j+1)k, n) - 1.  With cfg.storage LOCAL_ROPE (default) the
 * pool keeps K with RoPE applied at p_j (chunk-local positions); with PRE_ROPE it keeps K
 * before any positional embedding, as Sec. 3.3.1 stores the C2 tokens' KV.  V as is.
 *
 *   k, v     : MEANPOOL: device [L][n][Hkv][d] pre-RoPE per-token K/V.  Slot j is the mean
 *              of block j's rows divided by the block's true size (a stand-in for the
 *              trained extractor, adapted from the residual mean-pooling variant of
 *              Sec. 3.2.3).
 *              PROVIDED: device [L][m][Hkv][d] pre-RoPE slot K/V from an external
 *              extractor (the paper's C2 token K/V, Sec. 3.2.2); K is turned to p_j
 *              (LOCAL_ROPE) or kept as given (PRE_ROPE).
 *              STORED: host or device [L][m][Hkv][d] slots already in stored form (K at
 *              p_j under LOCAL_ROPE, K before RoPE under PRE_ROPE), copied verbatim -- the
 *              "load from host memory" step of Appendix C.
 *              HOST: the same stored form in pinned, device-mapped host memory, NOT copied:
 *              the chunk takes no pool slots and c2kv_compose reads it over the host link
 *              (load, re-rotation and gather in one pass).  The caller keeps the memory
 *              valid and unchanged until the chunk is freed.  ERR_ARG if k or v is not
 *              pinned (cudaHostAlloc / cudaHostRegister) or does not start on a 16-byte
 *              boundary; the whole L*m*Hkv*d span must lie in the pinned allocation.
 *   n_tokens : original chunk length n >= 1.
 *   ratio_k  : compression ratio k >= 1 (k = 1: uncompressed control).
 *   mode     : C2KV_MODE_*.
 *   chunk_id_out : receives the new chunk's id (>= 0).
 * The caller's buffers must stay valid until the stream reaches this call's work.
 * Errors: ERR_ARG, ERR_POOL_FULL (state unchanged), ERR_CUDA.
 */
c2kv_status c2kv_compress_chunk(c2kv_ctx* ctx, const void* k, const void* v, int32_t n_tokens,
                                int32_t ratio_k, int32_t mode, int32_t* chunk_id_out);

/* c2kv_free_chunk -- return a chunk's slots to the pool.  Composed caches already made
 * from it are unaffected (they hold copies).  Errors: ERR_BAD_CHUNK. */
c2kv_status c2kv_free_chunk(c2kv_ctx* ctx, int32_t chunk_id);

/* c2kv_chunk_info -- where a chunk lives in the pool.  Errors: ERR_BAD_CHUNK, ERR_ARG. */
c2kv_status c2kv_chunk_info(const c2kv_ctx* ctx, int32_t chunk_id, c2kv_chunk_desc* out);

/*
 * c2kv_compose -- the blending step B for a batch of requests (Sec. 3.2.4): each chunk
 * occurrence gets new positional embeddings for its placement -- offsets accumulate across
 * the concatenated segments and a compressed segment occupies its original span -- and
 * the slots are concatenated, without recomputation (Appendix C: load + position
 * reassignment + RoPE re-rotation).
 *
 * Occurrence i of request r (chunk c_i, n_i tokens, m_i slots, offset o_i) fills rows
 * row_base[r] + D_i + j, j < m_i, D_i = sum of earlier m, for every layer:
 *     K' = R(o_i) K_stored   (turn from p_j to o_i + p_j),   V' = V_stored,
 *     pos = o_i + p_j
 * under LOCAL_ROPE storage, and K' = RoPE(K_stored, o_i + p_j) under PRE_ROPE (the same
 * cache in exact arithmetic; each rounds K' to the storage dtype once per stored form).
 * With cfg.fixed_pos, pos = p_j and K' = K_stored (LOCAL_ROPE) or RoPE(K_stored, p_j).
 *
 *   batch           : number of requests B >= 1.
 *   req_ptr         : host [B + 1], CSR offsets into chunk_ids (req_ptr[0] = 0,
 *                     non-decreasing; a request may reuse no chunk).
 *   chunk_ids       : host [req_ptr[B]] chunk ids; duplicates allowed.
 *   positions       : host [req_ptr[B]] start offset o_i of each occurrence, or NULL for
 *                     o_0 = 0, o_{i+1} = o_i + n_i within each request.  Must satisfy
 *                     o_0 >= 0 and o_{i+1} >= o_i + n_i (gaps allowed: room for a static /
 *                     system prompt, Sec. 4.1), else ERR_POSITIONS.
 *   suffix_capacity : rows reserved after each request's slots for its suffix tokens.
 *   out             : receives a library-owned cache; each request's region starts at a
 *                     multiple of 128 rows and holds round_up(S_r + suffix_capacity, 128)
 *                     rows.
 * Errors: ERR_ARG, ERR_BAD_CHUNK, ERR_POSITIONS, ERR_NOMEM, ERR_CUDA.
 */
c2kv_status c2kv_compose(c2kv_ctx* ctx, int32_t batch, const int32_t* req_ptr,
                         const int32_t* chunk_ids, const int32_t* positions,
                         int32_t suffix_capacity, c2kv_cache** out);

/* c2kv_cache_info -- pointers and per-request metadata of a composed cache. */
c2kv_status c2kv_cache_info(const c2kv_cache* cache, c2kv_cache_desc* out);

/*
 * c2kv_attend -- the inference step F over [KV_total; x_q] (Sec. 2.2) with the model's
 * standard attention operator (Sec. 3.2.2): for each request r, suffix token t sits at
 * position L_r + t; its Q and K are RoPE'd there, its K/V written into the cache rows
 * right after the S_r composed slots, and
 *     O[t, h] = softmax_j( Q_t,h . K_j,h/G / sqrt(d) ) V_j,h/G     over keys j <= S_r + t
 * (every composed slot visible; causal inside the suffix; G = Hq / Hkv, query head h uses
 * KV head h / G).
 *
 *   layer    : layer index, or -1 for all layers in one launch.
 *   q        : [Lq][B][n_suffix][Hq][d] pre-RoPE queries (Lq = L if layer == -1, else 1).
 *   k_suf, v_suf : [Lq][B][n_suffix][Hkv][d] pre-RoPE suffix K, V.
 *   n_suffix : suffix tokens per request, 1 <= n_suffix <= the cache's suffix_capacity.
 *   out      : [Lq][B][n_suffix][Hq][d] attention output (context dtype).
 *   lse      : [Lq][B][Hq][n_suffix] fp32 natural-log softmax normaliser, or NULL.
 * q, k_suf, v_suf, out and lse are device memory or pinned host memory (page-locked and
 * mapped, e.g. cudaHostAlloc); host tensors are copied through device scratch on the
 * context's stream, in and out of the call.  The call is idempotent: it always writes the
 * suffix at rows S_r .. S_r + n_suffix - 1.
 * Errors: ERR_ARG (also for a tensor the GPU cannot address), ERR_STATE (cache from another
 * context), ERR_NOMEM, ERR_CUDA.
 */
c2kv_status c2kv_attend(c2kv_ctx* ctx, c2kv_cache* cache, int32_t layer, const void* q,
                        const void* k_suf, const void* v_suf, int32_t n_suffix, void* out,
                        float* lse);

/*
 * c2kv_compose_attend -- blending and inference in one call: the same result as
 *     c2kv_compose(ctx, batch, req_ptr, chunk_ids, positions, suffix_capacity, cache_out)
 *     c2kv_attend(ctx, *cache_out, -1, q, k_suf, v_suf, n_suffix, out, lse)
 * (the composed cache, its positions, the suffix rows, O and lse), for every layer.  On
 * the tensor-core route (bf16, d 128) with every chunk in the device pool, at most 32
 * requests, at most 128 chunk occurrences and LOCAL_ROPE storage, one fused kernel does all of it: the
 * attention reads each composed slot straight from the pool, turns K by its occurrence's
 * offset in shared memory (Sec. 3.2.4 re-rotation), turns the queries and the suffix keys by
 * their positions, and writes the composed cache as it goes, so the cache is written once
 * and never read back (a small kernel before it evaluates the suffix positions' angles).
 * Otherwise compose and attention run one after the other, the suffix preparation beside
 * compose on a second stream (it writes only rows compose does not; in turn while a trace
 * is on); with chunks in host memory and two or more layers, the layers go in groups so
 * that reading one group over the host link overlaps the attention of the previous one (on
 * a second stream).  Either way the call's work ends on the context's stream.  The context's `fuse` setting chooses (C2KV_FUSE_*): by
 * default the fused kernel runs when each (layer, request, KV head) has one pair of query
 * tiles.  The cache is returned as by c2kv_compose (release it with c2kv_cache_release) and
 * serves later c2kv_decode / c2kv_attend calls.
 *
 *   batch, req_ptr, chunk_ids, positions, suffix_capacity : as c2kv_compose.
 *   q, k_suf, v_suf, n_suffix, out, lse : as c2kv_attend with layer = -1 (device or pinned
 *                host memory; with chunks in host memory the host tensors move per layer
 *                group, each group's suffix in while it is composed and its output out while
 *                the next group is read); 1 <= n_suffix <= suffix_capacity.
 *   cache_out : receives the composed cache.
 * Errors: the union of c2kv_compose's and c2kv_attend's; on error no cache is returned.
 */
c2kv_status c2kv_compose_attend(c2kv_ctx* ctx, int32_t batch, const int32_t* req_ptr,
                                const int32_t* chunk_ids, const int32_t* positions,
                                int32_t suffix_capacity, const void* q, const void* k_suf,
                                const void* v_suf, int32_t n_suffix, void* out, float* lse,
                                c2kv_cache** cache_out);

/*
 * c2kv_attend_noalloc -- the same computation and arguments as c2kv_attend, for callers
 * that cannot let the library allocate device memory while they run: for example a
 * serving engine that reserves all of HBM for its own cache pool at start-up and treats
 * any later allocation as an error, or a host runtime whose allocator must own every
 * device byte.  The paper has no counterpart; this is a deployment variant.
 *
 * c2kv_attend takes its scratch (the suffix queries after RoPE, which the attention
 * kernels read) from the context's memory pool.  This call instead uses one fixed 16 MiB
 * array that the library defines in device memory; it calls no allocator at all.
 *   - Refused with C2KV_ERR_ARG (before anything is enqueued) when the rotated queries,
 *     Lq * batch * n_suffix * Hq * head_dim * element size bytes, exceed 16 MiB; split
 *     such a call by layer or by requests.
 *   - c2kv_create looks up the array's device address on the context's device and loads
 *     every kernel this call can launch there, so the array (and the kernels' code) is
 *     reserved when the context is made, not at the first call: under CUDA's lazy module
 *     loading that first call would otherwise be the moment device memory is taken.  Every
 *     GPU on which a context is created holds the 16 MiB until the process exits.
 *   - The current device must be the context's device (ERR_STATE otherwise).
 *   - All calls on a device share the array: calls whose GPU work overlaps (other
 *     streams, other contexts on the same device) race on it.  It keeps the last call's
 *     contents; nothing in it needs to start at zero.
 *   - q, k_suf, v_suf, out and lse may be device memory or pinned, mapped host memory, as
 *     for c2kv_attend; host tensors are read and written in place over the CPU-GPU link
 *     (c2kv_attend copies them through scratch instead).  Memory the GPU cannot address is
 *     refused with ERR_ARG.
 *   - Unlike c2kv_attend, it never splits a work unit's key range over several CTAs (the
 *     split partials would need scratch), so a single layer of a small batch leaves most
 *     SMs idle; and its launches are not recorded by the trace (c2kv_profile_*).
 * Errors: as c2kv_attend, plus ERR_ARG for the size limit.
 */
c2kv_status c2kv_attend_noalloc(c2kv_ctx* ctx, c2kv_cache* cache, int32_t layer,
                                const void* q, const void* k_suf, const void* v_suf,
                                int32_t n_suffix, void* out, float* lse);

/*
 * c2kv_decode -- one generation step after the suffix (the decode phase that follows the
 * first token; time between tokens): for each request r the new token, suffix index
 * steps[r], sits at position L_r + steps[r].  Its Q and K are RoPE'd there, its K/V written
 * to cache row S_r + steps[r], and
 *     O[h] = softmax_j( Q_h . K_j,h/G / sqrt(d) ) V_j,h/G      over keys j <= S_r + steps[r]
 * (every composed slot and suffix rows 0 .. steps[r]; G = Hq / Hkv).  This is the same
 * operator as c2kv_attend for one query row (Sec. 3.2.2).  Rows S_r .. S_r + steps[r] - 1
 * must already hold the earlier suffix tokens (written by c2kv_attend or earlier decode
 * calls); the library does not track which rows were written.  A later c2kv_attend zeroes
 * the rows after its own suffix up to the next 128-row boundary, decoded rows included.
 *
 *   layer : layer index, or -1 for all layers in one launch.
 *   q     : device [Lq][B][Hq][d] pre-RoPE query of the new token (Lq = L if layer == -1).
 *   k_new, v_new : device [Lq][B][Hkv][d] pre-RoPE K, V of the new token.
 *   steps : host int32[B], 0 <= steps[r] < the cache's suffix_capacity.
 *   out   : device [Lq][B][Hq][d] attention output (context dtype).
 *   lse   : device [Lq][B][Hq] fp32 natural-log softmax normaliser, or NULL.
 * q, k_new, v_new, out and lse must be device (or managed) memory: anything else is
 * refused with ERR_ARG before anything is enqueued.
 * The key range of each (layer, request, KV head) is split over several CTAs and merged
 * exactly (log-sum-exp; on the tensor-core route by the last split of each unit, inside the
 * kernel); the split buffer comes from the context's memory pool.  With bf16
 * and d = 128 the step runs on the tensor-core attention kernel (the new token as a one-row
 * query tile) when (layers x requests x KV heads) fits one CTA per SM or a request holds
 * 4096 keys or more, else on a CUDA-core decode kernel (C2KV_ATTN_TC forces the former,
 * C2KV_ATTN_SIMT the latter).
 * The tensor-core route reads whole 128-row key tiles, so it zeroes the rows after the new
 * one up to the next 128-row boundary that no earlier call on this cache has written or
 * zeroed (never rows an earlier c2kv_attend or c2kv_decode wrote).
 * Errors: ERR_ARG, ERR_STATE (cache from another context), ERR_UNSUPPORTED (head layout the
 * decode kernel does not take: G = Hq/Hkv in {1,2,4,8,16}, d in {64,128}, G*d <= 1024, and
 * G <= 8 for bf16), ERR_NOMEM, ERR_CUDA.
 */
c2kv_status c2kv_decode(c2kv_ctx* ctx, c2kv_cache* cache, int32_t layer, const void* q,
                        const void* k_new, const void* v_new, const int32_t* steps, void* out,
                        float* lse);

/*
 * c2kv_extract_attention -- one attention layer of the C2 Extractor's forward over a chunk
 * under the Structured Information Flow mask (Sec. 3.3).  The sequence is the n document
 * tokens followed by the m = ceil(n/k) C2 tokens, [x_0 .. x_{n-1}; c_0 .. c_{m-1}]
 * (Sec. 3.3.1); document token t sits at position t, C2 token c_j at the position of the
 * last token of its block B(j) = [jk, min((j+1)k, n)).  Q and K are RoPE'd there and
 *     O[t, h] = softmax_u( Q_t,h . K_u,h/G / sqrt(d) + M[t, u] ) V_u,h/G
 * with the mask (Sec. 3.3.2):
 *   - a document token sees document tokens 0..t only (so its output is the frozen model's);
 *   - c_j sees the document tokens of B(j) and of the sink block, and c_0 .. c_j.
 * The sink block, B(0) in the paper's 1-based numbering, is read as the first block
 * [0, min(k, n)).  The trained C2 embeddings and QKV projections that produce q, k, v for
 * the C2 tokens are the caller's; this is the attention operator they feed.  On the
 * tensor-core route (bf16, d 128) the C2 rows' launch runs on the context's second stream
 * beside the document rows' attention; the call's work ends on the context's stream.
 *
 *   n_layers : layers in the tensors (each processed independently).
 *   q        : device [n_layers][n + m][Hq][d] pre-RoPE queries.
 *   k, v     : device [n_layers][n + m][Hkv][d] pre-RoPE keys, values.
 *   n_tokens : n >= 1;  ratio_k : k >= 1.
 *   out      : device [n_layers][n + m][Hq][d] (context dtype).
 *   lse      : device [n_layers][Hq][n + m] fp32 natural-log normaliser, or NULL.
 * q, k, v, out and lse must be device (or managed) memory: anything else is refused with
 * ERR_ARG before anything is enqueued.
 * Errors: ERR_ARG, ERR_UNSUPPORTED (d not 64 or 128), ERR_NOMEM, ERR_CUDA.
 */
c2kv_status c2kv_extract_attention(c2kv_ctx* ctx, int32_t n_layers, const void* q, const void* k,
                                   const void* v, int32_t n_tokens, int32_t ratio_k, void* out,
                                   float* lse);

/* c2kv_cache_release -- free a composed cache (stream-ordered). */
c2kv_status c2kv_cache_release(c2kv_ctx* ctx, c2kv_cache* cache);

/* c2kv_sync -- wait for the context's stream; returns ERR_DEVICE_BOUNDS if any kernel's
 * bounds check refused an index since the last sync (the refused access was skipped), or
 * ERR_CUDA for a CUDA error. */
c2kv_status c2kv_sync(c2kv_ctx* ctx);

/* c2kv_last_error -- message for the last failing call on this context ("" if none).
 * Valid until the next call on the context.  NULL ctx gives the last create() failure. */
const char* c2kv_last_error(const c2kv_ctx* ctx);

/*
 * Tracing: per-kernel device time.  While enabled, each kernel launch the library makes
 * (compose, compress, suffix RoPE/append, attention, decode, extraction) is bracketed by
 * CUDA events on the context's stream.  Enabling creates a stock of events up front, so a
 * traced call only records them.  c2kv_profile_read synchronizes the stream and returns,
 * per kind, the mean device time of the launches recorded since the previous read (or
 * since enabling), then forgets them.  Kinds index the arrays:
 */
#define C2KV_PROF_COMPOSE  0
#define C2KV_PROF_COMPRESS 1
#define C2KV_PROF_SUFFIX   2   /* suffix RoPE + append + pad zeroing */
#define C2KV_PROF_ATTN     3   /* the attention kernel alone */
#define C2KV_PROF_COMBINE  4   /* merge of key-range splits (when attention was split) */
#define C2KV_PROF_DECODE   5   /* decode attention (with the merge of its splits) */
#define C2KV_PROF_EXTRACT  6   /* SIF-masked extraction attention (RoPE + attention) */
#define C2KV_PROF_FUSED    7   /* fused compose + attention kernel (c2kv_compose_attend) */
#define C2KV_PROF_KINDS    8
c2kv_status c2kv_profile_enable(c2kv_ctx* ctx, int32_t on);
/* mean_ms[C2KV_PROF_KINDS] receives mean milliseconds (0 where none), launches[] the
 * counts; either may be NULL. */
c2kv_status c2kv_profile_read(c2kv_ctx* ctx, float* mean_ms, int32_t* launches);

/* c2kv_inject_fault -- host-side fault injection for tests.  what = 1: the next compose
 * writes one out-of-range pool slot index into its slot map, which the compose kernel's
 * bounds check must refuse (reported by c2kv_sync as ERR_DEVICE_BOUNDS).  what = 0 clears. */
c2kv_status c2kv_inject_fault(c2kv_ctx* ctx, int32_t what);

#ifdef __cplusplus
}
#endif

#endif /* C2KV_H */
