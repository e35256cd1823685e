// c2kv_attend_noalloc: suffix attention that allocates no device memory.
//
// Some callers cannot let a library call cudaMalloc (or allocate from a stream-ordered
// pool) once they are running: a serving engine that reserves all of HBM for its own
// KV-cache pool at start-up and treats any later allocation as a failure, a host runtime
// whose own allocator must own every device byte, or a latency-critical loop that must
// never wait on the driver's allocator.  For them this entry point takes its only scratch
// buffer -- the suffix queries after RoPE, which the attention kernels read as their Q
// operand -- from a fixed array in device memory that the library defines at file scope,
// instead of the context's memory pool used by c2kv_attend.
//
// Contract (also in include/c2kv.h):
//   * the array holds kNoAllocScratchBytes (16 MiB); requests whose rotated queries need
//     more (layers * batch * n_suffix * Hq * head_dim * element size) are refused with
//     C2KV_ERR_ARG before anything is enqueued;
//   * c2kv_create looks the array's device address up (cudaGetSymbolAddress, with the
//     context's device current) and loads every kernel this call can launch: under CUDA's
//     lazy module loading the first use of a module is when its device memory (static
//     arrays, code) is taken, and that must not be this call.  Every GPU on which a context
//     is created holds the array until the process exits;
//   * the current device must be the context's (the address belongs to that device);
//   * every call on a device shares the one array: two calls whose work overlaps on the
//     GPU (different streams, or different contexts on one device) race on it.  The array
//     keeps the last call's contents; nothing in it needs to start at zero, because each
//     call writes every rotated query row it later reads;
//   * suffix tensors in pinned, mapped host memory are read and written in place (there is
//     no scratch to stage them through); memory the GPU cannot address is refused;
//   * a work unit's key range is never split over several CTAs (that needs scratch for the
//     partials), and the launches are not traced.
#include <initializer_list>

#include "c2kv.h"
#include "internal.cuh"

namespace {

constexpr size_t kNoAllocScratchBytes = size_t(16) << 20;

static __device__ __align__(256) unsigned char g_attend_scratch[kNoAllocScratchBytes];

c2kv_status refuse(c2kv_ctx* ctx, c2kv_status code, const char* msg) {
    return c2kv::set_last_error(ctx, code, msg);
}

}  // namespace

namespace c2kv {

cudaError_t noalloc_prepare(int dtype, int d, bool tc, void** scratch) {
    *scratch = nullptr;
    void* p = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&p, g_attend_scratch);
    if (e == cudaSuccess) e = preload_suffix_kernels(dtype, d);
    if (e == cudaSuccess) e = tc ? preload_attn_tc_kernels() : preload_attn_simt_kernels(dtype, d);
    if (e != cudaSuccess) return e;
    *scratch = p;
    return cudaSuccess;
}

}  // namespace c2kv

extern "C" c2kv_status c2kv_attend_noalloc(c2kv_ctx* ctx, c2kv_cache* cache, int32_t layer,
                                           const void* q, const void* k_suf, const void* v_suf,
                                           int32_t n_suffix, void* out, float* lse) {
    if (!ctx) return C2KV_ERR_ARG;
    c2kv::AttendView v{};
    if (!c2kv::attend_view(ctx, cache, &v))
        return refuse(ctx, C2KV_ERR_STATE, "attend_noalloc: cache not owned by this context");
    if (!q || !k_suf || !v_suf || !out)
        return refuse(ctx, C2KV_ERR_ARG, "attend_noalloc: null pointer");
    const auto misaligned = [](const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) != 0; };
    if (misaligned(q, 16) || misaligned(k_suf, 16) || misaligned(v_suf, 16) || misaligned(out, 16) ||
        misaligned(lse, 4))
        return refuse(ctx, C2KV_ERR_ARG, "attend_noalloc: misaligned tensor pointer");
    for (const void* p : {q, k_suf, v_suf, static_cast<const void*>(out), static_cast<const void*>(lse)})
        if (c2kv::mem_kind(p) == c2kv::MemKind::kUnknown)
            return refuse(ctx, C2KV_ERR_ARG,
                          "attend_noalloc: tensor in memory the GPU cannot address (neither device "
                          "nor pinned, mapped host memory)");
    if (layer < -1 || layer >= v.layers)
        return refuse(ctx, C2KV_ERR_ARG, "attend_noalloc: bad layer");
    if (n_suffix < 1 || n_suffix > v.suffix_capacity)
        return refuse(ctx, C2KV_ERR_ARG, "attend_noalloc: n_suffix outside [1, suffix_capacity]");
    const int32_t lq = layer < 0 ? v.layers : 1;
    const int32_t layer0 = layer < 0 ? 0 : layer;
    const int32_t B = v.batch;
    const size_t eb = v.dtype == C2KV_DTYPE_BF16 ? 2 : 4;
    const size_t q_bytes = (size_t)lq * B * n_suffix * v.n_q_heads * v.head_dim * eb;
    if (q_bytes > kNoAllocScratchBytes)
        return refuse(ctx, C2KV_ERR_ARG,
                      "attend_noalloc: the rotated queries need more than the library's fixed "
                      "16 MiB scratch array (layers * batch * n_suffix * Hq * head_dim * "
                      "element size); split the call by layer or by request batch, or use "
                      "c2kv_attend");
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        (void)cudaGetLastError();
        return refuse(ctx, C2KV_ERR_CUDA, "attend_noalloc: cannot read the current device");
    }
    if (dev != v.device || v.noalloc_scratch == nullptr)
        return refuse(ctx, C2KV_ERR_STATE,
                      "attend_noalloc: the current device is not the context's device");
    void* const q_rot = v.noalloc_scratch;
    cudaError_t e = cudaSuccess;
    const bool use_tc = v.attn_impl != C2KV_ATTN_SIMT &&
                        c2kv::attn_tc_supported(v.dtype, v.head_dim, v.n_q_heads, v.n_kv_heads);
    for (int32_t b0 = 0; e == cudaSuccess && b0 < B; b0 += c2kv::kMaxReq) {
        const int32_t nb = B - b0 < c2kv::kMaxReq ? B - b0 : c2kv::kMaxReq;
        c2kv::SuffixParams s{};
        s.q = q;
        s.k = k_suf;
        s.v = v_suf;
        s.q_rot = q_rot;
        s.cache_k = v.cache_k;
        s.cache_v = v.cache_v;
        s.pos = v.pos;
        s.rows = v.rows;
        s.layer0 = layer0;
        s.lq = lq;
        s.batch = nb;
        s.batch_total = B;
        s.b0 = b0;
        s.sq = n_suffix;
        s.hq = v.n_q_heads;
        s.hkv = v.n_kv_heads;
        s.pad_rows = 1;
        s.rope = v.turns;
        for (int32_t i = 0; i < nb; ++i) {
            s.req[i] = c2kv::ReqParam{v.row_base[b0 + i], v.n_slots[b0 + i], v.l_req[b0 + i], 0};
            s.pad_from[i] = v.n_slots[b0 + i] + n_suffix;
        }
        e = c2kv::launch_suffix_prep(s, v.dtype, v.head_dim, v.stream);
        if (e != cudaSuccess) break;
        c2kv::AttnParams a{};
        a.q_rot = q_rot;
        a.cache_k = v.cache_k;
        a.cache_v = v.cache_v;
        a.out = out;
        a.lse = lse;
        a.err = v.err;
        a.rows = v.rows;
        a.layer0 = layer0;
        a.lq = lq;
        a.batch = nb;
        a.batch_total = B;
        a.b0 = b0;
        a.sq = n_suffix;
        a.hq = v.n_q_heads;
        a.hkv = v.n_kv_heads;
        a.scale_log2 = (float)(1.4426950408889634 / __builtin_sqrt((double)v.head_dim));
        a.pairs_per_cta = v.attn_pairs;
        for (int32_t i = 0; i < nb; ++i) a.req[i] = s.req[i];
        e = use_tc ? c2kv::launch_attn_tc(a, v.stream)
                   : c2kv::launch_attn_simt(a, v.dtype, v.head_dim, v.stream);
    }
    if (e != cudaSuccess) {
        (void)cudaGetLastError();
        return refuse(ctx, C2KV_ERR_CUDA, "attend_noalloc: kernel launch failed");
    }
    c2kv::note_suffix_written(cache, layer0, lq, n_suffix);
    c2kv::set_last_error(ctx, C2KV_OK, "");
    return C2KV_OK;
}
