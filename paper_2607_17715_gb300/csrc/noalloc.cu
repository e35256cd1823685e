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
//   * every GPU on which the library's device code is loaded holds the array until the
//     process exits;
//   * the first call on a device looks the array's device address up (cudaGetSymbolAddress,
//     with that device current) and caches it; make that first call before any stream
//     capture;
//   * every call on a device shares the one array: two calls whose work overlaps on the
//     GPU (different streams, or different contexts on one device) race on it.  The array
//     keeps the last call's contents; nothing in it needs to start at zero, because each
//     call writes every rotated query row it later reads.
#include <mutex>

#include "c2kv.h"
#include "internal.cuh"

namespace {

constexpr size_t kNoAllocScratchBytes = size_t(16) << 20;
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_attend_scratch[kNoAllocScratchBytes];

std::mutex g_scratch_mu;
void* g_scratch_addr[kMaxDevices] = {};

// Device address of g_attend_scratch on the current device (looked up once per device).
cudaError_t scratch_address(void** out) {
    *out = nullptr;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_scratch_mu);
    if (!g_scratch_addr[dev]) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_attend_scratch);
        if (e != cudaSuccess) return e;
        g_scratch_addr[dev] = p;
    }
    *out = g_scratch_addr[dev];
    return cudaSuccess;
}

c2kv_status refuse(c2kv_ctx* ctx, c2kv_status code, const char* msg) {
    return c2kv::set_last_error(ctx, code, msg);
}

}  // namespace

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
    void* q_rot = nullptr;
    cudaError_t e = scratch_address(&q_rot);
    if (e != cudaSuccess) {
        (void)cudaGetLastError();
        return refuse(ctx, C2KV_ERR_CUDA, "attend_noalloc: cannot resolve the scratch array");
    }
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
        for (int32_t i = 0; i < nb; ++i)
            s.req[i] = c2kv::ReqParam{v.row_base[b0 + i], v.n_slots[b0 + i], v.l_req[b0 + i], 0};
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
        for (int32_t i = 0; i < nb; ++i) a.req[i] = s.req[i];
        e = use_tc ? c2kv::launch_attn_tc(a, v.stream)
                   : c2kv::launch_attn_simt(a, v.dtype, v.head_dim, v.stream);
    }
    if (e != cudaSuccess) {
        (void)cudaGetLastError();
        return refuse(ctx, C2KV_ERR_CUDA, "attend_noalloc: kernel launch failed");
    }
    c2kv::set_last_error(ctx, C2KV_OK, "");
    return C2KV_OK;
}
