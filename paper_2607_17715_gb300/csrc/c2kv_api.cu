// Host side of the C2KV library: the C ABI declared in include/c2kv.h.
//
// Owns the device chunk pool (a slot arena with a first-fit free list), validates every
// request before anything is enqueued (so a failing call leaves no trace), packs the small
// per-call metadata (chunk occurrences, per-request row layout, RoPE frequencies as 0.64
// fixed-point turns) into the kernels' parameter blocks -- no host-to-device copy per call
// -- and launches the kernels on the context's stream.  Composed caches and per-call
// scratch come from a context-owned stream-ordered memory pool.
#include "c2kv.h"
#include "internal.cuh"

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdint>
#include <cstdio>
#include <cstring>
#include <initializer_list>
#include <map>
#include <new>
#include <string>
#include <vector>


namespace {

constexpr int64_t kTileRows = 128;   // composed-cache request regions align to this

struct Chunk {
    int32_t n = 0, k = 0, m = 0, base = 0;
    bool live = false;
    bool host = false;                  // registered in host memory (C2KV_MODE_HOST)
    const void* host_k = nullptr;       // device-accessible addresses of the host slots
    const void* host_v = nullptr;
};

thread_local std::string g_create_error;

}  // namespace

struct c2kv_cache {
    c2kv_ctx* owner = nullptr;
    int32_t batch = 0, layers = 0;
    int64_t rows = 0;
    void* k = nullptr;
    void* v = nullptr;
    int32_t* pos = nullptr;        // device [rows]
    std::vector<int32_t> row_base, n_slots, l_req, capacity;
    // [layer][request]: rows of the request's region known to hold finite values (written or
    // zeroed) from its first row on; the tensor-core decode zeroes the rest of the key tile
    // that holds its new row before it reads it
    std::vector<int32_t> clean_to;
    int32_t suffix_capacity = 0;
};

struct c2kv_ctx {
    c2kv_config cfg{};
    cudaStream_t stream = nullptr;
    int device = 0;
    int eb = 2;
    void* pool_k = nullptr;
    void* pool_v = nullptr;
    std::vector<Chunk> chunks;
    std::map<int32_t, int32_t> free_ranges;   // start -> length
    std::string err;
    int32_t* d_err = nullptr;
    cudaMemPool_t mempool = nullptr;
    std::vector<c2kv_cache*> caches;
    int32_t inject = 0;
    int sms = 148;
    void* noalloc_scratch = nullptr;   // c2kv_attend_noalloc's fixed array on this device
    // per-unit counters of the tensor-core attention's in-kernel split merge: zero between
    // launches (each unit's last split sets its counter back), cleared again after a device error
    uint32_t* tickets = nullptr;
    size_t tickets_cap = 0;
    c2kv::RopeTurns turns{};
    // second stream and events of the pipelined compose + attend (host-resident chunks)
    cudaStream_t aux = nullptr;
    std::vector<cudaEvent_t> aux_ev;
    // tracing (c2kv_profile_enable): event pairs around launches, by kind
    bool prof = false;
    struct ProfRec { int kind; cudaEvent_t a, b; };
    std::vector<ProfRec> prof_recs;
    std::vector<cudaEvent_t> prof_free;
};

namespace {

c2kv_status fail(c2kv_ctx* ctx, c2kv_status code, const char* fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof(buf), fmt, ap);
    va_end(ap);
    if (ctx) ctx->err = buf;
    else g_create_error = buf;
    return code;
}

c2kv_status cuda_fail(c2kv_ctx* ctx, cudaError_t e, const char* what) {
    (void)cudaGetLastError();   // a non-sticky failure must not leak into later calls
    return fail(ctx, e == cudaErrorMemoryAllocation ? C2KV_ERR_NOMEM : C2KV_ERR_CUDA,
                "%s: %s", what, cudaGetErrorString(e));
}

int64_t row_elems(const c2kv_ctx* c) { return (int64_t)c->cfg.n_kv_heads * c->cfg.head_dim; }

cudaError_t pool_alloc(c2kv_ctx* c, void** p, size_t bytes) {
    *p = nullptr;
    if (bytes == 0) bytes = 256;
    return cudaMallocFromPoolAsync(p, bytes, c->mempool, c->stream);
}

void pool_free(c2kv_ctx* c, void* p) {
    if (p) cudaFreeAsync(p, c->stream);
}

// At least n zeroed split-merge counters (grown rarely: the old array may still be in use by
// work on the stream, so the stream drains first).
cudaError_t tickets_ready(c2kv_ctx* c, size_t n) {
    if (n <= c->tickets_cap) return cudaSuccess;
    const size_t cap = std::max<size_t>({n, 2 * c->tickets_cap, 4096});
    cudaError_t e = cudaStreamSynchronize(c->stream);
    if (e != cudaSuccess) return e;
    if (c->tickets) cudaFree(c->tickets);
    c->tickets = nullptr;
    c->tickets_cap = 0;
    void* p = nullptr;
    e = cudaMalloc(&p, cap * sizeof(uint32_t));
    // ordered on the context's stream, which need not synchronise with the legacy stream
    if (e == cudaSuccess) e = cudaMemsetAsync(p, 0, cap * sizeof(uint32_t), c->stream);
    if (e != cudaSuccess) {
        if (p) cudaFree(p);
        return e;
    }
    c->tickets = static_cast<uint32_t*>(p);
    c->tickets_cap = cap;
    return cudaSuccess;
}

// RoPE frequency i = theta^(-2i/d) as a fraction of a turn in 0.64 fixed point, from
// long-double arithmetic (the kernels' phase accumulator; see internal.cuh).
void make_turns(c2kv::RopeTurns* t, double theta, int d) {
    const long double two_pi = 6.283185307179586476925286766559005768L;
    for (int i = 0; i < c2kv::kMaxHalf; ++i) {
        if (i >= d / 2) {
            t->turn[i] = 0;
            continue;
        }
        const long double f = std::pow((long double)theta, -2.0L * i / d) / two_pi;
        t->turn[i] = (uint64_t)std::llround(std::ldexp(f, 64));
    }
}

bool take_range(c2kv_ctx* c, int32_t m, int32_t* base) {
    for (auto it = c->free_ranges.begin(); it != c->free_ranges.end(); ++it) {
        if (it->second >= m) {
            *base = it->first;
            const int32_t rest = it->second - m;
            const int32_t start = it->first + m;
            c->free_ranges.erase(it);
            if (rest > 0) c->free_ranges[start] = rest;
            return true;
        }
    }
    return false;
}

void give_range(c2kv_ctx* c, int32_t base, int32_t m) {
    if (m <= 0) return;
    auto it = c->free_ranges.emplace(base, m).first;
    auto next = std::next(it);
    if (next != c->free_ranges.end() && it->first + it->second == next->first) {
        it->second += next->second;
        c->free_ranges.erase(next);
    }
    if (it != c->free_ranges.begin()) {
        auto prev = std::prev(it);
        if (prev->first + prev->second == it->first) {
            prev->second += it->second;
            c->free_ranges.erase(it);
        }
    }
}

bool is_device_ptr(const void* p) {
    cudaPointerAttributes at{};
    if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    return at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged;
}

// Every tensor pointer is at least this aligned (16 bytes; lse arrays 4): the kernels move
// rows in 16-byte vectors and by TMA, and a misaligned vector access would fault.
bool aligned(const void* p, uintptr_t a = 16) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; }

using c2kv::MemKind;
using c2kv::mem_kind;

// Refuses (ERR_ARG) any of the tensors that is not device or managed memory: the calls whose
// kernels take only device tensors (decode, extraction).
c2kv_status require_device(c2kv_ctx* c, const char* what, std::initializer_list<const void*> ps) {
    for (const void* p : ps)
        if (mem_kind(p) != MemKind::kDevice)
            return fail(c, C2KV_ERR_ARG, "%s: tensors must be device memory (a pointer is host "
                                         "memory or memory the GPU cannot address)", what);
    return C2KV_OK;
}

bool own_cache(const c2kv_ctx* c, const c2kv_cache* cache) {
    return cache && std::find(c->caches.begin(), c->caches.end(), cache) != c->caches.end();
}

void destroy_cache(c2kv_ctx* c, c2kv_cache* cache) {
    pool_free(c, cache->k);
    pool_free(c, cache->v);
    pool_free(c, cache->pos);
    delete cache;
}

constexpr size_t kProfEvents = 1024;   // events made ready when tracing is enabled

cudaEvent_t prof_event(c2kv_ctx* c) {
    if (!c->prof_free.empty()) {
        cudaEvent_t e = c->prof_free.back();
        c->prof_free.pop_back();
        return e;
    }
    cudaEvent_t e = nullptr;
    if (cudaEventCreate(&e) != cudaSuccess) {
        (void)cudaGetLastError();
        return nullptr;
    }
    return e;
}

// Brackets the launches between begin() and end() with events when tracing is on.
struct ProfScope {
    c2kv_ctx* c;
    int kind;
    cudaEvent_t a = nullptr;
    // deferred: the start event is recorded by start(), which a launcher calls through its
    // Hook once its host-side preparation is done
    ProfScope(c2kv_ctx* ctx, int k, bool deferred = false) : c(ctx), kind(k) {
        if (!deferred) start();
    }
    void start() {
        if (!a && c->prof && (a = prof_event(c)) != nullptr) cudaEventRecord(a, c->stream);
    }
    c2kv::Hook hook() {
        return c2kv::Hook{[](void* self) { static_cast<ProfScope*>(self)->start(); }, this};
    }
    ~ProfScope() {
        if (!a) return;
        cudaEvent_t b = prof_event(c);
        if (!b) {
            c->prof_free.push_back(a);
            return;
        }
        cudaEventRecord(b, c->stream);
        c->prof_recs.push_back({kind, a, b});
    }
};

}  // namespace

extern "C" {

int32_t c2kv_abi_version(void) { return C2KV_ABI_VERSION; }

const char* c2kv_last_error(const c2kv_ctx* ctx) {
    return ctx ? ctx->err.c_str() : g_create_error.c_str();
}

c2kv_status c2kv_create(const c2kv_config* cfg, void* stream, c2kv_ctx** out) {
    try {
        if (!cfg || !out) return fail(nullptr, C2KV_ERR_ARG, "create: null cfg or out");
        *out = nullptr;
        const c2kv_config& f = *cfg;
        if (f.layers < 1 || f.n_q_heads < 1 || f.n_kv_heads < 1 || f.n_q_heads % f.n_kv_heads)
            return fail(nullptr, C2KV_ERR_ARG, "create: bad layer/head counts");
        if (f.head_dim != 64 && f.head_dim != 128)
            return fail(nullptr, C2KV_ERR_ARG, "create: head_dim must be 64 or 128");
        if (!(f.rope_theta > 1.0)) return fail(nullptr, C2KV_ERR_ARG, "create: rope_theta <= 1");
        if (f.dtype != C2KV_DTYPE_BF16 && f.dtype != C2KV_DTYPE_F32)
            return fail(nullptr, C2KV_ERR_DTYPE, "create: dtype must be BF16 or F32");
        if (f.pool_slots < 1) return fail(nullptr, C2KV_ERR_ARG, "create: pool_slots < 1");
        if (f.attn_impl < C2KV_ATTN_AUTO || f.attn_impl > C2KV_ATTN_TC)
            return fail(nullptr, C2KV_ERR_ARG, "create: bad attn_impl");
        if (f.attn_split < 0 || f.attn_split > 16)
            return fail(nullptr, C2KV_ERR_ARG, "create: attn_split outside [0, 16]");
        if (f.fuse < C2KV_FUSE_AUTO || f.fuse > C2KV_FUSE_ALWAYS)
            return fail(nullptr, C2KV_ERR_ARG, "create: bad fuse setting");
        if (f.storage != C2KV_STORAGE_LOCAL_ROPE && f.storage != C2KV_STORAGE_PRE_ROPE)
            return fail(nullptr, C2KV_ERR_ARG, "create: bad storage setting");
        if (f.attn_pairs < 0) return fail(nullptr, C2KV_ERR_ARG, "create: attn_pairs < 0");
        if (f.attn_impl == C2KV_ATTN_TC &&
            !c2kv::attn_tc_supported(f.dtype, f.head_dim, f.n_q_heads, f.n_kv_heads))
            return fail(nullptr, C2KV_ERR_UNSUPPORTED,
                        "create: tensor-core attention needs bf16, head_dim 128, Hq/Hkv in {1,2,4,8,16}");
        auto* c = new c2kv_ctx();
        c->cfg = f;
        c->stream = static_cast<cudaStream_t>(stream);
        c->eb = f.dtype == C2KV_DTYPE_BF16 ? 2 : 4;
        cudaError_t e = cudaGetDevice(&c->device);
        if (e == cudaSuccess) e = cudaDeviceGetAttribute(&c->sms, cudaDevAttrMultiProcessorCount, c->device);
        const size_t pool_bytes = (size_t)f.layers * (size_t)f.pool_slots * (size_t)row_elems(c) * c->eb;
        if (e == cudaSuccess) e = cudaMalloc(&c->pool_k, pool_bytes);
        if (e == cudaSuccess) e = cudaMalloc(&c->pool_v, pool_bytes);
        if (e == cudaSuccess) e = cudaMalloc(&c->d_err, sizeof(int32_t));
        if (e == cudaSuccess) e = cudaMemset(c->d_err, 0, sizeof(int32_t));
        if (e == cudaSuccess) {
            // c2kv_attend_noalloc's scratch array and kernels, reserved now rather than at
            // its first call (lazy module loading)
            const bool tc = f.attn_impl != C2KV_ATTN_SIMT &&
                            c2kv::attn_tc_supported(f.dtype, f.head_dim, f.n_q_heads, f.n_kv_heads);
            e = c2kv::noalloc_prepare(f.dtype, f.head_dim, tc, &c->noalloc_scratch);
        }
        if (e == cudaSuccess) {
            cudaMemPoolProps props{};
            props.allocType = cudaMemAllocationTypePinned;
            props.location.type = cudaMemLocationTypeDevice;
            props.location.id = c->device;
            e = cudaMemPoolCreate(&c->mempool, &props);
            if (e == cudaSuccess) {
                uint64_t keep = UINT64_MAX;
                e = cudaMemPoolSetAttribute(c->mempool, cudaMemPoolAttrReleaseThreshold, &keep);
            }
        }
        if (e != cudaSuccess) {
            cuda_fail(nullptr, e, "create");
            c2kv_destroy(c);
            return e == cudaErrorMemoryAllocation ? C2KV_ERR_NOMEM : C2KV_ERR_CUDA;
        }
        c->free_ranges[0] = f.pool_slots;
        make_turns(&c->turns, f.rope_theta, f.head_dim);
        *out = c;
        return C2KV_OK;
    } catch (const std::bad_alloc&) {
        return fail(nullptr, C2KV_ERR_NOMEM, "create: host allocation failed");
    } catch (...) {
        return fail(nullptr, C2KV_ERR_ARG, "create: unexpected failure");
    }
}

c2kv_status c2kv_destroy(c2kv_ctx* c) {
    if (!c) return C2KV_OK;
    try {
        if (c->stream || c->pool_k) cudaStreamSynchronize(c->stream);
        for (c2kv_cache* cache : c->caches) destroy_cache(c, cache);
        c->caches.clear();
        cudaStreamSynchronize(c->stream);
        for (auto& r : c->prof_recs) {
            cudaEventDestroy(r.a);
            cudaEventDestroy(r.b);
        }
        for (cudaEvent_t e : c->prof_free) cudaEventDestroy(e);
        if (c->aux) {
            cudaStreamSynchronize(c->aux);
            cudaStreamDestroy(c->aux);
        }
        for (cudaEvent_t e : c->aux_ev) cudaEventDestroy(e);
        if (c->mempool) cudaMemPoolDestroy(c->mempool);
        if (c->pool_k) cudaFree(c->pool_k);
        if (c->pool_v) cudaFree(c->pool_v);
        if (c->d_err) cudaFree(c->d_err);
        if (c->tickets) cudaFree(c->tickets);
        delete c;
        return C2KV_OK;
    } catch (...) {
        return C2KV_ERR_STATE;
    }
}

c2kv_status c2kv_set_stream(c2kv_ctx* c, void* stream) {
    if (!c) return C2KV_ERR_ARG;
    c->stream = static_cast<cudaStream_t>(stream);
    c->err.clear();
    return C2KV_OK;
}

c2kv_status c2kv_compress_chunk(c2kv_ctx* c, const void* k, const void* v, int32_t n_tokens,
                                int32_t ratio_k, int32_t mode, int32_t* chunk_id_out) {
    if (!c) return C2KV_ERR_ARG;
    try {
        c->err.clear();
        if (!k || !v || !chunk_id_out) return fail(c, C2KV_ERR_ARG, "compress: null pointer");
        if (!aligned(k) || !aligned(v)) return fail(c, C2KV_ERR_ARG, "compress: k, v must be 16-byte aligned");
        if (n_tokens < 1 || ratio_k < 1) return fail(c, C2KV_ERR_ARG, "compress: need n >= 1, k >= 1");
        if (mode != C2KV_MODE_MEANPOOL && mode != C2KV_MODE_PROVIDED && mode != C2KV_MODE_STORED &&
            mode != C2KV_MODE_HOST)
            return fail(c, C2KV_ERR_ARG, "compress: bad mode %d", mode);
        if (mode == C2KV_MODE_HOST) {
            // no copy: keep the device-accessible addresses of the caller's pinned slots
            const void* dk = nullptr;
            const void* dv = nullptr;
            for (int w = 0; w < 2; ++w) {
                cudaPointerAttributes at{};
                const void* p = w ? v : k;
                if (cudaPointerGetAttributes(&at, p) != cudaSuccess || at.type != cudaMemoryTypeHost ||
                    at.devicePointer == nullptr) {
                    (void)cudaGetLastError();
                    return fail(c, C2KV_ERR_ARG, "compress: HOST mode needs pinned, device-mapped host memory");
                }
                if (reinterpret_cast<uintptr_t>(at.devicePointer) % 16 != 0)
                    return fail(c, C2KV_ERR_ARG, "compress: HOST mode slots must start on a 16-byte boundary");
                (w ? dv : dk) = at.devicePointer;
            }
            int32_t id = -1;
            for (size_t i = 0; i < c->chunks.size(); ++i)
                if (!c->chunks[i].live) { id = (int32_t)i; break; }
            if (id < 0) {
                c->chunks.emplace_back();
                id = (int32_t)c->chunks.size() - 1;
            }
            Chunk& ch = c->chunks[id];
            ch = Chunk{};
            ch.n = n_tokens;
            ch.k = ratio_k;
            ch.m = (int32_t)(((int64_t)n_tokens + ratio_k - 1) / ratio_k);
            ch.base = -1;
            ch.live = true;
            ch.host = true;
            ch.host_k = dk;
            ch.host_v = dv;
            *chunk_id_out = id;
            return C2KV_OK;
        }
        if (mode != C2KV_MODE_STORED && (!is_device_ptr(k) || !is_device_ptr(v)))
            return fail(c, C2KV_ERR_ARG, "compress: MEANPOOL/PROVIDED inputs must be device memory");
        const int32_t m = (int32_t)(((int64_t)n_tokens + ratio_k - 1) / ratio_k);
        int32_t base = 0;
        if (!take_range(c, m, &base))
            return fail(c, C2KV_ERR_POOL_FULL, "compress: no free range of %d slots", m);
        const size_t rb = (size_t)row_elems(c) * c->eb;
        cudaError_t e = cudaSuccess;
        if (mode == C2KV_MODE_STORED) {
            const size_t dpitch = (size_t)c->cfg.pool_slots * rb;
            char* dk = static_cast<char*>(c->pool_k) + (size_t)base * rb;
            char* dv = static_cast<char*>(c->pool_v) + (size_t)base * rb;
            e = cudaMemcpy2DAsync(dk, dpitch, k, (size_t)m * rb, (size_t)m * rb, c->cfg.layers,
                                  cudaMemcpyDefault, c->stream);
            if (e == cudaSuccess)
                e = cudaMemcpy2DAsync(dv, dpitch, v, (size_t)m * rb, (size_t)m * rb,
                                      c->cfg.layers, cudaMemcpyDefault, c->stream);
        } else {
            c2kv::CompressParams a{};
            a.in_k = k;
            a.in_v = v;
            a.pool_k = c->pool_k;
            a.pool_v = c->pool_v;
            a.pool_slots = c->cfg.pool_slots;
            a.slot_base = base;
            a.m = m;
            a.n = n_tokens;
            a.k = ratio_k;
            a.one_row = mode == C2KV_MODE_PROVIDED ? 1 : 0;
            a.rows_in = mode == C2KV_MODE_PROVIDED ? m : n_tokens;
            a.layers = c->cfg.layers;
            a.hkv = c->cfg.n_kv_heads;
            a.turn = c->cfg.storage == C2KV_STORAGE_LOCAL_ROPE ? 1 : 0;
            a.rope = c->turns;
            ProfScope prof_compress(c, C2KV_PROF_COMPRESS);
            e = c2kv::launch_compress(a, c->cfg.dtype, c->cfg.head_dim, c->stream);
        }
        if (e != cudaSuccess) {
            give_range(c, base, m);
            return cuda_fail(c, e, "compress");
        }
        int32_t id = -1;
        for (size_t i = 0; i < c->chunks.size(); ++i)
            if (!c->chunks[i].live) { id = (int32_t)i; break; }
        if (id < 0) {
            c->chunks.emplace_back();
            id = (int32_t)c->chunks.size() - 1;
        }
        Chunk& ch = c->chunks[id];
        ch = Chunk{};
        ch.n = n_tokens;
        ch.k = ratio_k;
        ch.m = m;
        ch.base = base;
        ch.live = true;
        *chunk_id_out = id;
        return C2KV_OK;
    } catch (const std::bad_alloc&) {
        return fail(c, C2KV_ERR_NOMEM, "compress: host allocation failed");
    }
}

c2kv_status c2kv_free_chunk(c2kv_ctx* c, int32_t id) {
    if (!c) return C2KV_ERR_ARG;
    c->err.clear();
    if (id < 0 || id >= (int32_t)c->chunks.size() || !c->chunks[id].live)
        return fail(c, C2KV_ERR_BAD_CHUNK, "free_chunk: unknown chunk %d", id);
    Chunk& ch = c->chunks[id];
    if (!ch.host) give_range(c, ch.base, ch.m);
    ch.live = false;
    return C2KV_OK;
}

c2kv_status c2kv_chunk_info(const c2kv_ctx* c, int32_t id, c2kv_chunk_desc* out) {
    if (!c || !out) return C2KV_ERR_ARG;
    if (id < 0 || id >= (int32_t)c->chunks.size() || !c->chunks[id].live) return C2KV_ERR_BAD_CHUNK;
    const Chunk& ch = c->chunks[id];
    const size_t rb = (size_t)row_elems(c) * c->eb;
    out->n_tokens = ch.n;
    out->ratio_k = ch.k;
    out->n_slots = ch.m;
    out->slot_base = ch.base;
    if (ch.host) {
        out->k = const_cast<void*>(ch.host_k);
        out->v = const_cast<void*>(ch.host_v);
        out->layer_stride = (int64_t)ch.m * row_elems(c);
    } else {
        out->k = static_cast<char*>(c->pool_k) + (size_t)ch.base * rb;
        out->v = static_cast<char*>(c->pool_v) + (size_t)ch.base * rb;
        out->layer_stride = (int64_t)c->cfg.pool_slots * row_elems(c);
    }
    return C2KV_OK;
}

}  // extern "C"

namespace {

// Validates a compose request and lays out its rows: on success `*out` is a new cache with
// its device buffers allocated (not yet registered with the context) and `occ` holds every
// occurrence's parameters.  On failure nothing is allocated.
c2kv_status compose_plan(c2kv_ctx* c, int32_t batch, const int32_t* req_ptr, const int32_t* chunk_ids,
                         const int32_t* positions, int32_t suffix_capacity, c2kv_cache** out,
                         std::vector<c2kv::OccParam>& occ) {
    if (!out || !req_ptr || batch < 1) return fail(c, C2KV_ERR_ARG, "compose: bad batch/out/req_ptr");
    *out = nullptr;
    if (suffix_capacity < 0) return fail(c, C2KV_ERR_ARG, "compose: suffix_capacity < 0");
    if (req_ptr[0] != 0) return fail(c, C2KV_ERR_ARG, "compose: req_ptr[0] != 0");
    for (int32_t r = 0; r < batch; ++r)
        if (req_ptr[r + 1] < req_ptr[r]) return fail(c, C2KV_ERR_ARG, "compose: req_ptr decreases");
    const int32_t n_occ = req_ptr[batch];
    if (n_occ > 0 && !chunk_ids) return fail(c, C2KV_ERR_ARG, "compose: null chunk_ids");

    // Validate everything and lay out the rows before touching the device.
    occ.assign((size_t)n_occ, c2kv::OccParam{});
    auto* cache = new c2kv_cache();
    cache->owner = c;
    cache->batch = batch;
    cache->layers = c->cfg.layers;
    cache->suffix_capacity = suffix_capacity;
    cache->row_base.resize(batch);
    cache->n_slots.resize(batch);
    cache->l_req.resize(batch);
    cache->capacity.resize(batch);
    int64_t row = 0;
    for (int32_t r = 0; r < batch; ++r) {
        int64_t slots = 0, prev_end = 0;
        for (int32_t i = req_ptr[r]; i < req_ptr[r + 1]; ++i) {
            const int32_t id = chunk_ids[i];
            if (id < 0 || id >= (int32_t)c->chunks.size() || !c->chunks[id].live) {
                delete cache;
                return fail(c, C2KV_ERR_BAD_CHUNK, "compose: unknown chunk %d (occurrence %d)", id, i);
            }
            const Chunk& ch = c->chunks[id];
            const int64_t o = positions ? positions[i] : prev_end;
            if (o < 0 || o < prev_end) {
                delete cache;
                return fail(c, C2KV_ERR_POSITIONS,
                            "compose: request %d occurrence %d starts at %lld before %lld", r, i,
                            (long long)o, (long long)prev_end);
            }
            prev_end = o + ch.n;
            if (prev_end > INT32_MAX) {
                delete cache;
                return fail(c, C2KV_ERR_POSITIONS, "compose: positions exceed int32");
            }
            c2kv::OccParam& rec = occ[i];
            rec.src_base = ch.base;
            rec.dest_row = (int32_t)(row + slots);
            rec.delta = c->cfg.fixed_pos ? 0 : (int32_t)o;
            rec.n = ch.n;
            rec.k = ch.k;
            rec.m = ch.m;
            rec.tile_base = 0;
            rec.host = ch.host ? 1 : 0;
            rec.host_k = ch.host_k;
            rec.host_v = ch.host_v;
            slots += ch.m;
        }
        const int64_t cap = (slots + suffix_capacity + kTileRows - 1) / kTileRows * kTileRows;
        if (row + cap > INT32_MAX) {
            delete cache;
            return fail(c, C2KV_ERR_ARG, "compose: batch too large");
        }
        cache->row_base[r] = (int32_t)row;
        cache->n_slots[r] = (int32_t)slots;
        cache->l_req[r] = (int32_t)prev_end;
        cache->capacity[r] = (int32_t)cap;
        row += cap;
    }
    cache->rows = row;
    cache->clean_to.assign((size_t)cache->layers * batch, 0);
    for (int32_t l = 0; l < cache->layers; ++l)
        for (int32_t r = 0; r < batch; ++r) cache->clean_to[(size_t)l * batch + r] = cache->n_slots[r];
    if (c->inject == 1 && n_occ > 0) {
        occ[0].src_base = c->cfg.pool_slots + 7;   // refused by the kernels' bounds checks
        c->inject = 0;
    }

    const size_t kv_bytes = (size_t)c->cfg.layers * (size_t)std::max<int64_t>(row, 1) *
                            (size_t)row_elems(c) * c->eb;
    const size_t pos_bytes = (size_t)std::max<int64_t>(row, 1) * sizeof(int32_t);
    cudaError_t e = pool_alloc(c, &cache->k, kv_bytes);
    if (e == cudaSuccess) e = pool_alloc(c, &cache->v, kv_bytes);
    if (e == cudaSuccess) e = pool_alloc(c, reinterpret_cast<void**>(&cache->pos), pos_bytes);
    if (e != cudaSuccess) {
        destroy_cache(c, cache);
        return cuda_fail(c, e, "compose: cache allocation");
    }
    *out = cache;
    return C2KV_OK;
}

// Composed slots per compose tile: the largest power of two up to kComposeTile that still
// gives about six CTAs per SM over the launch's slots and layers, so that a small launch
// (one layer of a few thousand slots) spreads over every SM instead of leaving a partial
// wave of large tiles, while a large one keeps the 16-slot tiles that amortise each CTA's
// angle table.
int32_t compose_tile_slots(const c2kv_ctx* c, int64_t slots, int32_t n_layers, int max_ctas) {
    if (max_ctas > 0) return c2kv::kComposeTile;    // a capped grid walks tiles anyway
    int32_t t = c2kv::kComposeTile;
    while (t > 2 && (slots + t - 1) / t * n_layers < 6LL * c->sms) t /= 2;
    return t;
}

// Slots per tile of the bulk-copy compose kernel: at most 16 KB of K rows (the stage then
// holds 32 KB of K and V, six of them in flight per SM), halved while the launch would give
// fewer than two tiles per SM, so that a small launch still spreads over the SMs (each tile
// costs its CTA about a microsecond of fixed work, so smaller tiles than that lose more than
// they balance: on the one-layer long70b shape, 8-slot tiles took 14.8-15.1 us against
// 15.7-15.8 us for 4-slot ones, and a threshold of eight tiles per SM 18.7 us).
int32_t compose_bulk_tile_slots(const c2kv_ctx* c, const std::vector<c2kv::OccParam>& occ, int32_t g0,
                                int32_t g1, int32_t n_layers) {
    const int64_t row_bytes = (int64_t)c->cfg.n_kv_heads * c->cfg.head_dim * c->eb;
    int32_t t = 1;
    while (t * 2 <= c2kv::kComposeBulkTile && (int64_t)t * 2 * row_bytes <= 16384) t *= 2;
    auto tiles = [&](int32_t ts) {
        int64_t n = 0;
        for (int32_t i = g0; i < g1; ++i) n += (occ[i].m + ts - 1) / ts;
        return n * n_layers;
    };
    while (t > 1 && tiles(t) < 2LL * c->sms) t /= 2;
    return t;
}

// The compose kernel over every occurrence: one launch per group of at most kMaxOcc
// occurrences, all layers at once; the bulk-copy kernel when every chunk of the group is in
// the device pool and the grid is not capped.
cudaError_t compose_launch(c2kv_ctx* c, const c2kv_cache* cache, const std::vector<c2kv::OccParam>& occ,
                           int32_t layer0 = 0, int32_t n_layers = -1, int max_ctas = 0) {
    const int32_t n_occ = (int32_t)occ.size();
    if (n_layers < 0) n_layers = c->cfg.layers;
    cudaError_t e = cudaSuccess;
    ProfScope prof_compose(c, C2KV_PROF_COMPOSE, true);
    for (int32_t g0 = 0; e == cudaSuccess && g0 < n_occ; g0 += c2kv::kMaxOcc) {
        const int32_t g1 = std::min(n_occ, g0 + c2kv::kMaxOcc);
        int64_t slots = 0;
        bool bulk = max_ctas == 0;
        for (int32_t i = g0; i < g1; ++i) {
            slots += occ[i].m;
            bulk = bulk && !occ[i].host;
        }
        const int32_t ts = bulk ? compose_bulk_tile_slots(c, occ, g0, g1, n_layers)
                                : compose_tile_slots(c, slots, n_layers, max_ctas);
        c2kv::ComposeParams pr{};
        pr.pool_k = c->pool_k;
        pr.pool_v = c->pool_v;
        pr.out_k = cache->k;
        pr.out_v = cache->v;
        pr.pos = cache->pos;
        pr.err = c->d_err;
        pr.pool_slots = c->cfg.pool_slots;
        pr.rows = cache->rows;
        pr.hkv = c->cfg.n_kv_heads;
        pr.layer0 = layer0;
        pr.tile_slots = ts;
        pr.bulk = bulk ? 1 : 0;
        pr.pre_rope = c->cfg.storage == C2KV_STORAGE_PRE_ROPE ? 1 : 0;
        pr.rope = c->turns;
        int32_t tiles = 0;
        for (int32_t i = g0; i < g1; ++i) {
            if (occ[i].m == 0) continue;
            c2kv::OccParam rec = occ[i];
            rec.tile_base = tiles;
            pr.occ[pr.n_occ++] = rec;
            tiles += (rec.m + ts - 1) / ts;
        }
        pr.n_tiles = tiles;
        e = c2kv::launch_compose(pr, c->cfg.dtype, c->cfg.head_dim, n_layers, c->stream, max_ctas,
                                 prof_compose.hook());
    }
    return e;
}

// After a suffix of n_suffix tokens over layers [l0, l0 + n): every request's rows up to the
// 128-row edge after its suffix hold finite values (the suffix rows, then zeros).
void mark_suffix_clean(c2kv_cache* cache, int32_t l0, int32_t n, int32_t n_suffix) {
    for (int32_t l = l0; l < l0 + n; ++l)
        for (int32_t r = 0; r < cache->batch; ++r) {
            int32_t& ct = cache->clean_to[(size_t)l * cache->batch + r];
            const int64_t edge = ((int64_t)cache->n_slots[r] + n_suffix + kTileRows - 1) / kTileRows * kTileRows;
            ct = std::max<int32_t>(ct, (int32_t)std::min<int64_t>(edge, cache->capacity[r]));
        }
}

// Checks of an attend call's arguments that do not depend on the cache's contents.
c2kv_status attend_check(c2kv_ctx* c, const char* what, int32_t layer, const void* q, const void* k_suf,
                         const void* v_suf, int32_t n_suffix, int32_t suffix_capacity, void* out,
                         float* lse) {
    if (!q || !k_suf || !v_suf || !out) return fail(c, C2KV_ERR_ARG, "%s: null pointer", what);
    if (!aligned(q) || !aligned(k_suf) || !aligned(v_suf) || !aligned(out) || !aligned(lse, 4))
        return fail(c, C2KV_ERR_ARG, "%s: misaligned tensor pointer", what);
    for (const void* p : {q, k_suf, v_suf, static_cast<const void*>(out), static_cast<const void*>(lse)})
        if (mem_kind(p) == MemKind::kUnknown)
            return fail(c, C2KV_ERR_ARG, "%s: tensor in memory the GPU cannot address (neither device "
                                         "nor pinned, mapped host memory)", what);
    if (layer < -1 || layer >= c->cfg.layers) return fail(c, C2KV_ERR_ARG, "%s: bad layer %d", what, layer);
    if (n_suffix < 1 || n_suffix > suffix_capacity)
        return fail(c, C2KV_ERR_ARG, "%s: n_suffix %d outside [1, %d]", what, n_suffix, suffix_capacity);
    return C2KV_OK;
}

// The suffix kernel's parameters for requests b0 .. b0 + nb - 1 of a cache.
c2kv::SuffixParams suffix_params(const c2kv_ctx* c, const c2kv_cache* cache, int32_t layer0, int32_t lq,
                                 const void* q, const void* k_suf, const void* v_suf, int32_t n_suffix,
                                 void* q_rot, int32_t b0, int32_t nb) {
    c2kv::SuffixParams s{};
    s.q = q;
    s.k = k_suf;
    s.v = v_suf;
    s.q_rot = q_rot;
    s.cache_k = cache->k;
    s.cache_v = cache->v;
    s.pos = cache->pos;
    s.rows = cache->rows;
    s.layer0 = layer0;
    s.lq = lq;
    s.batch = nb;
    s.batch_total = cache->batch;
    s.b0 = b0;
    s.sq = n_suffix;
    s.hq = c->cfg.n_q_heads;
    s.hkv = c->cfg.n_kv_heads;
    s.pad_rows = 1;
    s.rope = c->turns;
    for (int32_t i = 0; i < nb; ++i) {
        s.req[i] = c2kv::ReqParam{cache->row_base[b0 + i], cache->n_slots[b0 + i], cache->l_req[b0 + i], 0};
        s.pad_from[i] = cache->n_slots[b0 + i] + n_suffix;
    }
    return s;
}

// The suffix preparation of every request alone (suffix RoPE into q_rot, the suffix rows and
// the zero rows up to the tile edge into the cache), on the context's stream.
cudaError_t suffix_run(c2kv_ctx* c, const c2kv_cache* cache, int32_t layer0, int32_t lq, const void* q,
                       const void* k_suf, const void* v_suf, int32_t n_suffix, void* q_rot) {
    cudaError_t e = cudaSuccess;
    for (int32_t b0 = 0; e == cudaSuccess && b0 < cache->batch; b0 += c2kv::kMaxReq) {
        const int32_t nb = std::min<int32_t>(c2kv::kMaxReq, cache->batch - b0);
        const c2kv::SuffixParams s = suffix_params(c, cache, layer0, lq, q, k_suf, v_suf, n_suffix, q_rot, b0, nb);
        ProfScope prof_suffix(c, C2KV_PROF_SUFFIX);
        e = c2kv::launch_suffix_prep(s, c->cfg.dtype, c->cfg.head_dim, c->stream);
    }
    return e;
}

// Suffix preparation and attention of a cache (arguments already checked).  With `fused`,
// the cache is not written yet: the fused kernel reads the composed slots from the pool and
// the suffix from k_suf / v_suf, turns the queries itself, and writes the whole cache
// (tensor-core route, every layer, one launch).  With `q_rot_ready`, the suffix preparation
// has already run (suffix_run) into that buffer: only attention is launched.
cudaError_t attend_run(c2kv_ctx* c, c2kv_cache* cache, int32_t layer0, int32_t lq, const void* q,
                       const void* k_suf, const void* v_suf, int32_t n_suffix, void* out, float* lse,
                       const c2kv::FusedSpec* fused, void* q_rot_ready = nullptr) {
    const int32_t B = cache->batch;
    const bool use_tc =
        c->cfg.attn_impl != C2KV_ATTN_SIMT &&
        c2kv::attn_tc_supported(c->cfg.dtype, c->cfg.head_dim, c->cfg.n_q_heads, c->cfg.n_kv_heads);
    if (fused && (!use_tc || layer0 != 0 || lq != c->cfg.layers || B > c2kv::kMaxReq))
        return cudaErrorInvalidValue;

    // scratch: the suffix queries after RoPE (the attention kernels' Q operand); the fused
    // kernel turns them in shared memory
    const size_t q_bytes = (size_t)lq * B * n_suffix * c->cfg.n_q_heads * c->cfg.head_dim * c->eb;
    void* q_rot = q_rot_ready;
    cudaError_t e = fused || q_rot_ready ? cudaSuccess : pool_alloc(c, &q_rot, q_bytes);
    if (e != cudaSuccess) return e;
    void* const q_rot_own = q_rot_ready ? nullptr : q_rot;    // freed here
    // Key-range split of the tensor-core attention: when its work units would leave most
    // SMs idle (a single layer of a small batch), each unit's key tiles are split and the
    // partials merged; at a wave or more the split only adds the merge.
    int32_t n_split = 1;
    float* part = nullptr;
    if (use_tc) {
        const int64_t units = c2kv::attn_tc_units(c->cfg.n_q_heads, c->cfg.n_kv_heads, n_suffix, lq, B);
        int32_t n_kv_max = 1;
        for (int32_t b = 0; b < B; ++b)
            n_kv_max = std::max<int32_t>(n_kv_max, (cache->n_slots[b] + n_suffix + 127) / 128);
        if (fused && fused->pairs_in_turn) {
            n_split = 1;             // one CTA runs every pair of its (layer, request, KV head)
        } else if (c->cfg.attn_split >= 1) {
            n_split = c->cfg.attn_split;
        } else if (2 * units <= c->sms) {
            // at most half of the SMs would have work: split toward one wave, keeping at
            // least 8 key tiles per split (below that the merge costs more than it saves)
            n_split = (int32_t)std::min<int64_t>(16, c->sms / units);
            n_split = std::max<int32_t>(1, std::min<int32_t>(n_split, n_kv_max / 8));
        }
        if (n_split > 1) {
            const size_t rows = (size_t)lq * B * n_suffix * c->cfg.n_q_heads;
            e = pool_alloc(c, reinterpret_cast<void**>(&part),
                           (size_t)n_split * rows * (c->cfg.head_dim + 1) * sizeof(float));
            // the plain kernel merges the splits itself (per-unit counters)
            if (e == cudaSuccess && !fused && n_split <= c2kv::kMaxMergeSplits)
                e = tickets_ready(c, (size_t)c2kv::attn_tc_units(c->cfg.n_q_heads, c->cfg.n_kv_heads, n_suffix,
                                                                 lq, std::min<int32_t>(B, c2kv::kMaxReq)));
            if (e != cudaSuccess) {
                pool_free(c, part);
                pool_free(c, q_rot_own);
                return e;
            }
        }
    }
    const bool merge_in_kernel = use_tc && !fused && n_split > 1 && n_split <= c2kv::kMaxMergeSplits;
    const size_t part_rows = (size_t)lq * B * n_suffix * c->cfg.n_q_heads;
    c2kv::AttnParams last{};
    for (int32_t b0 = 0; e == cudaSuccess && b0 < B; b0 += c2kv::kMaxReq) {
        const int32_t nb = std::min<int32_t>(c2kv::kMaxReq, B - b0);
        const c2kv::SuffixParams s = suffix_params(c, cache, layer0, lq, q, k_suf, v_suf, n_suffix, q_rot, b0, nb);
        c2kv::AttnParams a{};
        a.q_rot = fused ? q : q_rot;
        a.cache_k = cache->k;
        a.cache_v = cache->v;
        a.out = out;
        a.lse = lse;
        a.err = c->d_err;
        a.rows = cache->rows;
        a.layer0 = layer0;
        a.lq = lq;
        a.batch = nb;
        a.batch_total = B;
        a.b0 = b0;
        a.sq = n_suffix;
        a.hq = c->cfg.n_q_heads;
        a.hkv = c->cfg.n_kv_heads;
        a.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)c->cfg.head_dim));
        a.n_split = n_split;
        a.pairs_per_cta = c->cfg.attn_pairs;
        a.part_o = part;
        a.part_lse = part ? part + (size_t)n_split * part_rows * c->cfg.head_dim : nullptr;
        a.tickets = merge_in_kernel ? c->tickets : nullptr;
        for (int32_t i = 0; i < nb; ++i) a.req[i] = s.req[i];
        if (fused) {
            e = c2kv::prepare_attn_fused(a, *fused);
            if (e != cudaSuccess) break;
            ProfScope prof_fused(c, C2KV_PROF_FUSED, true);
            e = c2kv::launch_attn_fused(c->stream, prof_fused.hook());
        } else {
            if (!q_rot_ready) {
                ProfScope prof_suffix(c, C2KV_PROF_SUFFIX);
                e = c2kv::launch_suffix_prep(s, c->cfg.dtype, c->cfg.head_dim, c->stream);
            }
            if (e != cudaSuccess) break;
            // the suffix kernel's programmatic dependent (its start and set-up overlap that
            // kernel), unless a trace puts events between them or the suffix ran elsewhere
            a.dependent = !c->prof && !q_rot_ready ? 1 : 0;
            ProfScope prof_attn(c, C2KV_PROF_ATTN, use_tc);
            e = use_tc ? c2kv::launch_attn_tc(a, c->stream, prof_attn.hook())
                       : c2kv::launch_attn_simt(a, c->cfg.dtype, c->cfg.head_dim, c->stream);
        }
        last = a;
        last.dependent = !c->prof && !fused && use_tc ? 1 : 0;   // the merge: the attention's dependent
    }
    if (e == cudaSuccess && n_split > 1 && !merge_in_kernel) {   // one merge over every request's rows
        ProfScope prof_combine(c, C2KV_PROF_COMBINE);
        e = c2kv::launch_attn_combine(last, c->stream);
    }
    pool_free(c, part);
    pool_free(c, q_rot_own);
    return e;
}

// Makes `c->stream` another stream while it lives (a context is used from one host thread
// at a time), so that allocations, launches and the trace of a call land on that stream.
struct StreamSwap {
    c2kv_ctx* c;
    cudaStream_t saved;
    StreamSwap(c2kv_ctx* ctx, cudaStream_t s) : c(ctx), saved(ctx->stream) { c->stream = s; }
    ~StreamSwap() { c->stream = saved; }
};

// The context's second stream, and at least n events for forks to it and joins from it.
cudaError_t aux_ready(c2kv_ctx* c, size_t n) {
    if (!c->aux) {
        const cudaError_t e = cudaStreamCreateWithFlags(&c->aux, cudaStreamNonBlocking);
        if (e != cudaSuccess) {
            c->aux = nullptr;
            return e;
        }
    }
    while (c->aux_ev.size() < n) {
        cudaEvent_t ev = nullptr;
        const cudaError_t e = cudaEventCreateWithFlags(&ev, cudaEventDisableTiming);
        if (e != cudaSuccess) return e;
        c->aux_ev.push_back(ev);
    }
    return cudaSuccess;
}

// Compose + attend when chunks are read from host memory: compose is bound by the host link,
// so the layers go in groups.  The context's stream composes group g with a few CTAs (the
// link is the limit, and the other SMs stay free), and a second stream runs group g's suffix
// preparation and attention as soon as its composed rows are in, while group g + 1 is read.
// The call's work ends on the context's stream, and the second stream first waits for the
// work enqueued there before the call.
// Suffix tensors and outputs of a call, and where the kernels read and write them: the
// caller's buffers, or device scratch that copies fill and drain when the caller's are in
// pinned host memory (the kernels then touch device memory only, and each copy moves in one
// bulk transfer rather than as the kernels' small accesses across the link).
struct SuffixIO {
    const void* q;
    const void* k;
    const void* v;
    void* out;
    float* lse;
    bool staged = false;
    void* scratch = nullptr;
    size_t q_layer = 0, kv_layer = 0, lse_layer = 0;   // bytes per layer
};

cudaError_t suffix_io_open(c2kv_ctx* c, int32_t layers, int32_t B, int32_t n_suffix, const void* q,
                           const void* k_suf, const void* v_suf, void* out, float* lse, SuffixIO* io) {
    const size_t eb = (size_t)c->eb, d = (size_t)c->cfg.head_dim, L = (size_t)layers;
    io->q = q;
    io->k = k_suf;
    io->v = v_suf;
    io->out = out;
    io->lse = lse;
    io->q_layer = (size_t)B * n_suffix * c->cfg.n_q_heads * d * eb;
    io->kv_layer = (size_t)B * n_suffix * c->cfg.n_kv_heads * d * eb;
    io->lse_layer = (size_t)B * c->cfg.n_q_heads * n_suffix * sizeof(float);
    bool host = false;
    for (const void* p : {q, k_suf, v_suf, static_cast<const void*>(out), static_cast<const void*>(lse)})
        host = host || mem_kind(p) == MemKind::kHost;
    if (!host) return cudaSuccess;
    // q, out: q_layer each; k, v: kv_layer each; lse: lse_layer (16-byte aligned pieces)
    auto up = [](size_t x) { return (x + 255) / 256 * 256; };
    const size_t bytes = L * (2 * up(io->q_layer) + 2 * up(io->kv_layer) + (lse ? up(io->lse_layer) : 0));
    cudaError_t e = pool_alloc(c, &io->scratch, bytes);
    if (e != cudaSuccess) return e;
    char* p = static_cast<char*>(io->scratch);
    io->q = p;
    p += L * up(io->q_layer);
    io->k = p;
    p += L * up(io->kv_layer);
    io->v = p;
    p += L * up(io->kv_layer);
    io->out = p;
    p += L * up(io->q_layer);
    io->lse = lse ? reinterpret_cast<float*>(p) : nullptr;
    io->staged = true;    // each region holds its L layers at the caller's stride, then padding
    return cudaSuccess;
}

// Copy layers [l0, l0 + n) of the staged inputs in (on the context's current stream).
cudaError_t suffix_io_in(c2kv_ctx* c, const SuffixIO& io, const void* q, const void* k_suf,
                         const void* v_suf, int32_t l0, int32_t n) {
    if (!io.staged) return cudaSuccess;
    cudaError_t e = cudaSuccess;
    const size_t ql = io.q_layer, kl = io.kv_layer;
    auto cp = [&](const void* dst, const void* src, size_t bytes) {
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(const_cast<void*>(dst), src, bytes, cudaMemcpyDefault, c->stream);
    };
    cp(static_cast<const char*>(io.q) + l0 * ql, static_cast<const char*>(q) + l0 * ql, n * ql);
    cp(static_cast<const char*>(io.k) + l0 * kl, static_cast<const char*>(k_suf) + l0 * kl, n * kl);
    cp(static_cast<const char*>(io.v) + l0 * kl, static_cast<const char*>(v_suf) + l0 * kl, n * kl);
    return e;
}

// Copy layers [l0, l0 + n) of the staged outputs back (on the context's current stream).
cudaError_t suffix_io_out(c2kv_ctx* c, const SuffixIO& io, void* out, float* lse, int32_t l0, int32_t n) {
    if (!io.staged) return cudaSuccess;
    cudaError_t e = cudaMemcpyAsync(static_cast<char*>(out) + l0 * io.q_layer,
                                    static_cast<const char*>(io.out) + l0 * io.q_layer, n * io.q_layer,
                                    cudaMemcpyDefault, c->stream);
    if (e == cudaSuccess && lse)
        e = cudaMemcpyAsync(reinterpret_cast<char*>(lse) + l0 * io.lse_layer,
                            reinterpret_cast<const char*>(io.lse) + l0 * io.lse_layer, n * io.lse_layer,
                            cudaMemcpyDefault, c->stream);
    return e;
}

cudaError_t compose_attend_pipelined(c2kv_ctx* c, c2kv_cache* cache, const std::vector<c2kv::OccParam>& occ,
                                     const void* q, const void* k_suf, const void* v_suf,
                                     int32_t n_suffix, void* out, float* lse) {
    const int32_t L = c->cfg.layers;
    const int32_t groups = std::min<int32_t>(4, L);
    const int32_t per = (L + groups - 1) / groups;
    cudaError_t e = aux_ready(c, (size_t)groups + 2);
    if (e != cudaSuccess) return e;
    SuffixIO io;
    e = suffix_io_open(c, L, cache->batch, n_suffix, q, k_suf, v_suf, out, lse, &io);
    if (e != cudaSuccess) return e;
    const size_t lse_floats = io.lse_layer / sizeof(float);               // per layer
    e = cudaEventRecord(c->aux_ev[0], c->stream);                          // the caller's work
    if (e == cudaSuccess) e = cudaStreamWaitEvent(c->aux, c->aux_ev[0], 0);
    for (int32_t g = 0; e == cudaSuccess && g < groups; ++g) {
        const int32_t l0 = g * per;
        const int32_t nl = std::min(per, L - l0);
        if (nl <= 0) break;
        {   // the group's suffix slices in, on the second stream, while the group is composed
            StreamSwap on_aux(c, c->aux);
            e = suffix_io_in(c, io, q, k_suf, v_suf, l0, nl);
        }
        if (e != cudaSuccess) break;
        const int max_ctas = std::max(1, c->sms / (4 * nl));                // about a quarter of the SMs
        e = compose_launch(c, cache, occ, l0, nl, max_ctas);
        if (e == cudaSuccess) e = cudaEventRecord(c->aux_ev[1 + g], c->stream);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(c->aux, c->aux_ev[1 + g], 0);
        if (e != cudaSuccess) break;
        StreamSwap on_aux(c, c->aux);
        e = attend_run(c, cache, l0, nl, static_cast<const char*>(io.q) + l0 * io.q_layer,
                       static_cast<const char*>(io.k) + l0 * io.kv_layer,
                       static_cast<const char*>(io.v) + l0 * io.kv_layer, n_suffix,
                       static_cast<char*>(io.out) + l0 * io.q_layer, io.lse ? io.lse + l0 * lse_floats : nullptr,
                       nullptr);
        // the group's outputs back while the next group is read
        if (e == cudaSuccess) e = suffix_io_out(c, io, out, lse, l0, nl);
    }
    // the call ends on the context's stream, after everything on the second stream
    const cudaError_t e2 = cudaEventRecord(c->aux_ev[groups + 1], c->aux);
    if (e2 == cudaSuccess) cudaStreamWaitEvent(c->stream, c->aux_ev[groups + 1], 0);
    if (e != cudaSuccess || e2 != cudaSuccess) cudaStreamSynchronize(c->aux);
    pool_free(c, io.scratch);
    return e != cudaSuccess ? e : e2;
}

// Compose + attend from chunks in the pool when the step is not fused.  The suffix
// preparation writes only what compose does not (the turned queries, the suffix rows and the
// zero rows after them, their positions), so it runs on the second stream while compose runs
// on the context's stream, and attention follows both.
cudaError_t compose_attend_overlapped(c2kv_ctx* c, c2kv_cache* cache, const std::vector<c2kv::OccParam>& occ,
                                      const void* q, const void* k_suf, const void* v_suf, int32_t n_suffix,
                                      void* out, float* lse) {
    const int32_t L = c->cfg.layers;
    const size_t q_bytes = (size_t)L * cache->batch * n_suffix * c->cfg.n_q_heads * c->cfg.head_dim * c->eb;
    void* q_rot = nullptr;
    cudaError_t e = aux_ready(c, 2);
    if (e == cudaSuccess) e = pool_alloc(c, &q_rot, q_bytes);
    if (e != cudaSuccess) return e;
    e = cudaEventRecord(c->aux_ev[0], c->stream);       // the caller's work and q_rot's allocation
    if (e == cudaSuccess) e = cudaStreamWaitEvent(c->aux, c->aux_ev[0], 0);
    if (e == cudaSuccess) {
        StreamSwap on_aux(c, c->aux);
        e = suffix_run(c, cache, 0, L, q, k_suf, v_suf, n_suffix, q_rot);
    }
    cudaError_t e2 = cudaEventRecord(c->aux_ev[1], c->aux);
    if (e == cudaSuccess) e = compose_launch(c, cache, occ);
    if (e2 == cudaSuccess) e2 = cudaStreamWaitEvent(c->stream, c->aux_ev[1], 0);
    if (e == cudaSuccess && e2 == cudaSuccess)
        e = attend_run(c, cache, 0, L, q, k_suf, v_suf, n_suffix, out, lse, nullptr, q_rot);
    if (e != cudaSuccess || e2 != cudaSuccess) cudaStreamSynchronize(c->aux);
    pool_free(c, q_rot);
    return e != cudaSuccess ? e : e2;
}

}  // namespace

extern "C" {

c2kv_status c2kv_compose(c2kv_ctx* c, int32_t batch, const int32_t* req_ptr,
                         const int32_t* chunk_ids, const int32_t* positions,
                         int32_t suffix_capacity, c2kv_cache** out) {
    if (!c) return C2KV_ERR_ARG;
    try {
        c->err.clear();
        std::vector<c2kv::OccParam> occ;
        c2kv_cache* cache = nullptr;
        const c2kv_status st =
            compose_plan(c, batch, req_ptr, chunk_ids, positions, suffix_capacity, &cache, occ);
        if (st != C2KV_OK) return st;
        const cudaError_t e = compose_launch(c, cache, occ);
        if (e != cudaSuccess) {
            destroy_cache(c, cache);
            return cuda_fail(c, e, "compose");
        }
        c->caches.push_back(cache);
        *out = cache;
        return C2KV_OK;
    } catch (const std::bad_alloc&) {
        return fail(c, C2KV_ERR_NOMEM, "compose: host allocation failed");
    }
}

c2kv_status c2kv_compose_attend(c2kv_ctx* c, int32_t batch, const int32_t* req_ptr,
                                const int32_t* chunk_ids, const int32_t* positions,
                                int32_t suffix_capacity, const void* q, const void* k_suf,
                                const void* v_suf, int32_t n_suffix, void* out, float* lse,
                                c2kv_cache** cache_out) {
    if (!c) return C2KV_ERR_ARG;
    try {
        c->err.clear();
        if (!cache_out) return fail(c, C2KV_ERR_ARG, "compose_attend: null cache_out");
        *cache_out = nullptr;
        c2kv_status st = attend_check(c, "compose_attend", -1, q, k_suf, v_suf, n_suffix,
                                      suffix_capacity, out, lse);
        if (st != C2KV_OK) return st;
        std::vector<c2kv::OccParam> occ;
        c2kv_cache* cache = nullptr;
        st = compose_plan(c, batch, req_ptr, chunk_ids, positions, suffix_capacity, &cache, occ);
        if (st != C2KV_OK) return st;
        // The fused kernel takes pool-resident chunks on the tensor-core route, at most
        // kMaxFusedReq requests and at most kMaxFusedOcc occurrences; anything
        // else runs compose and then attention.  By default it runs only when one pair of
        // query tiles covers each (layer, request, KV head).  With more pairs, forcing it
        // (C2KV_FUSE_ALWAYS) runs them in turn in one CTA per (layer, request, KV head), the
        // last pair first (it composes the cache), the others over the cache; with forced
        // key-range splits each pair's CTA composes its own tiles instead.  Neither beat
        // composing once, then attending (batched: 106 us against 100 us of kernels).
        const int32_t grp = c->cfg.n_q_heads / std::max(1, c->cfg.n_kv_heads);
        const int64_t q_rows = (int64_t)n_suffix * grp;
        const int64_t tq = 128 / std::max(1, grp);
        const int64_t pairs = ((n_suffix + tq - 1) / tq + 1) / 2;
        const bool forced = c->cfg.fuse == C2KV_FUSE_ALWAYS;
        bool fuse = c->cfg.fuse != C2KV_FUSE_NEVER && (forced || q_rows <= 256) &&
                    c->cfg.attn_impl != C2KV_ATTN_SIMT &&
                    c2kv::attn_tc_supported(c->cfg.dtype, c->cfg.head_dim, c->cfg.n_q_heads,
                                            c->cfg.n_kv_heads) &&
                    batch <= c2kv::kMaxFusedReq && occ.size() <= (size_t)c2kv::kMaxFusedOcc;
        const bool pairs_in_turn = pairs > 1 && c->cfg.attn_split <= 1;
        bool host_chunks = false;
        for (const auto& o : occ) host_chunks = host_chunks || o.host;
        // PRE_ROPE slots turn by a position per slot, which the fused loaders' per-occurrence
        // angle tables do not hold: compose, then attend
        fuse = fuse && !host_chunks && c->cfg.storage == C2KV_STORAGE_LOCAL_ROPE;
        cudaError_t e = cudaSuccess;
        // suffix tensors and outputs in pinned host memory: copied through device scratch (the
        // pipelined route does this per layer group itself)
        SuffixIO io;
        const bool pipelined = !fuse && host_chunks && c->cfg.layers >= 2;
        if (!pipelined) {
            e = suffix_io_open(c, c->cfg.layers, batch, n_suffix, q, k_suf, v_suf, out, lse, &io);
            if (e == cudaSuccess) e = suffix_io_in(c, io, q, k_suf, v_suf, 0, c->cfg.layers);
            if (e != cudaSuccess) {
                pool_free(c, io.scratch);
                destroy_cache(c, cache);
                return cuda_fail(c, e, "compose_attend: staging the suffix");
            }
        }
        const void* q_d = pipelined ? q : io.q;
        const void* k_d = pipelined ? k_suf : io.k;
        const void* v_d = pipelined ? v_suf : io.v;
        void* out_d = pipelined ? out : io.out;
        float* lse_d = pipelined ? lse : io.lse;
        if (fuse) {
            static thread_local c2kv::FusedSpec f;   // 13 KB: kept off the stack
            f.pool_k = c->pool_k;
            f.pool_v = c->pool_v;
            f.pos = cache->pos;
            f.pool_slots = c->cfg.pool_slots;
            f.rope = c->turns;
            for (int32_t r = 0; r <= batch; ++r) f.req_occ[r] = req_ptr[r];
            for (size_t i = 0; i < occ.size(); ++i) {
                const int32_t r = (int32_t)(std::upper_bound(req_ptr, req_ptr + batch + 1, (int32_t)i) -
                                            req_ptr) - 1;
                f.occ[i] = c2kv::FusedOcc{occ[i].src_base, occ[i].dest_row - cache->row_base[r],
                                          occ[i].m, occ[i].delta, occ[i].n, occ[i].k};
            }
            // (cos, sin) per layer, occurrence and frequency, then per suffix token and frequency
            float2* occ_cs = nullptr;
            const size_t n_occ_cs = (size_t)c->cfg.layers * std::max<size_t>(occ.size(), 1) * 64;
            e = pool_alloc(c, reinterpret_cast<void**>(&occ_cs),
                           (n_occ_cs + (size_t)batch * n_suffix * 64) * sizeof(float2));
            if (e == cudaSuccess) {
                f.occ_cs = occ_cs;
                f.sfx_cs = occ_cs + n_occ_cs;
                f.pairs_in_turn = pairs_in_turn ? 1 : 0;
                f.k_suf = k_d;
                f.v_suf = v_d;
                e = attend_run(c, cache, 0, c->cfg.layers, q_d, k_d, v_d, n_suffix, out_d, lse_d, &f);
                pool_free(c, occ_cs);
            }
        } else if (pipelined) {
            e = compose_attend_pipelined(c, cache, occ, q, k_suf, v_suf, n_suffix, out, lse);
        } else if (!c->prof) {
            e = compose_attend_overlapped(c, cache, occ, q_d, k_d, v_d, n_suffix, out_d, lse_d);
        } else {    // traced: one kernel at a time, so that each recorded time is its kernel's own
            e = compose_launch(c, cache, occ);
            if (e == cudaSuccess)
                e = attend_run(c, cache, 0, c->cfg.layers, q_d, k_d, v_d, n_suffix, out_d, lse_d, nullptr);
        }
        if (e == cudaSuccess && !pipelined) e = suffix_io_out(c, io, out, lse, 0, c->cfg.layers);
        if (!pipelined) pool_free(c, io.scratch);
        if (e != cudaSuccess) {
            destroy_cache(c, cache);
            return cuda_fail(c, e, "compose_attend");
        }
        mark_suffix_clean(cache, 0, c->cfg.layers, n_suffix);
        c->caches.push_back(cache);
        *cache_out = cache;
        return C2KV_OK;
    } catch (const std::bad_alloc&) {
        return fail(c, C2KV_ERR_NOMEM, "compose_attend: host allocation failed");
    }
}

c2kv_status c2kv_cache_info(const c2kv_cache* cache, c2kv_cache_desc* out) {
    if (!cache || !out) return C2KV_ERR_ARG;
    out->batch = cache->batch;
    out->layers = cache->layers;
    out->rows = cache->rows;
    out->k = cache->k;
    out->v = cache->v;
    out->pos = cache->pos;
    out->row_base = cache->row_base.data();
    out->n_slots = cache->n_slots.data();
    out->l_req = cache->l_req.data();
    out->capacity = cache->capacity.data();
    out->suffix_capacity = cache->suffix_capacity;
    return C2KV_OK;
}

c2kv_status c2kv_attend(c2kv_ctx* c, c2kv_cache* cache, int32_t layer, const void* q,
                        const void* k_suf, const void* v_suf, int32_t n_suffix, void* out,
                        float* lse) {
    if (!c) return C2KV_ERR_ARG;
    try {
        c->err.clear();
        if (!own_cache(c, cache)) return fail(c, C2KV_ERR_STATE, "attend: cache not owned by this context");
        const c2kv_status st =
            attend_check(c, "attend", layer, q, k_suf, v_suf, n_suffix, cache->suffix_capacity, out, lse);
        if (st != C2KV_OK) return st;
        const int32_t lq = layer < 0 ? c->cfg.layers : 1;
        SuffixIO io;    // suffix tensors and outputs in pinned host memory: staged through scratch
        cudaError_t e = suffix_io_open(c, lq, cache->batch, n_suffix, q, k_suf, v_suf, out, lse, &io);
        if (e == cudaSuccess) e = suffix_io_in(c, io, q, k_suf, v_suf, 0, lq);
        if (e == cudaSuccess)
            e = attend_run(c, cache, layer < 0 ? 0 : layer, lq, io.q, io.k, io.v, n_suffix, io.out, io.lse,
                           nullptr);
        if (e == cudaSuccess) e = suffix_io_out(c, io, out, lse, 0, lq);
        pool_free(c, io.scratch);
        if (e != cudaSuccess) return cuda_fail(c, e, "attend");
        mark_suffix_clean(cache, layer < 0 ? 0 : layer, lq, n_suffix);
        return C2KV_OK;
    } catch (const std::bad_alloc&) {
        return fail(c, C2KV_ERR_NOMEM, "attend: host allocation failed");
    }
}

c2kv_status c2kv_decode(c2kv_ctx* c, c2kv_cache* cache, int32_t layer, const void* q,
                        const void* k_new, const void* v_new, const int32_t* steps, void* out,
                        float* lse) {
    if (!c) return C2KV_ERR_ARG;
    try {
        c->err.clear();
        if (!own_cache(c, cache)) return fail(c, C2KV_ERR_STATE, "decode: cache not owned by this context");
        if (!q || !k_new || !v_new || !steps || !out) return fail(c, C2KV_ERR_ARG, "decode: null pointer");
        if (!aligned(q) || !aligned(k_new) || !aligned(v_new) || !aligned(out) || !aligned(lse, 4))
            return fail(c, C2KV_ERR_ARG, "decode: misaligned tensor pointer");
        if (const c2kv_status st = require_device(c, "decode", {q, k_new, v_new, out, lse})) return st;
        if (layer < -1 || layer >= c->cfg.layers) return fail(c, C2KV_ERR_ARG, "decode: bad layer %d", layer);
        if (!c2kv::decode_supported(c->cfg.dtype, c->cfg.head_dim, c->cfg.n_q_heads, c->cfg.n_kv_heads))
            return fail(c, C2KV_ERR_UNSUPPORTED, "decode: head layout not supported");
        const int32_t B = cache->batch;
        int32_t n_keys_max = 1;
        for (int32_t b = 0; b < B; ++b) {
            if (steps[b] < 0 || steps[b] >= cache->suffix_capacity)
                return fail(c, C2KV_ERR_ARG, "decode: steps[%d] = %d outside [0, %d)", b, steps[b],
                            cache->suffix_capacity);
            n_keys_max = std::max<int32_t>(n_keys_max, cache->n_slots[b] + steps[b] + 1);
        }
        if (B == 0) return C2KV_OK;
        const int32_t lq = layer < 0 ? c->cfg.layers : 1;
        const int32_t layer0 = layer < 0 ? 0 : layer;
        const int32_t hq = c->cfg.n_q_heads, hkv = c->cfg.n_kv_heads, d = c->cfg.head_dim;
        const int64_t units = (int64_t)hkv * lq * std::min<int32_t>(B, c2kv::kMaxReq);
        // bf16, d 128: the tensor-core attention kernel with the new token as a one-row
        // suffix at suffix index steps[r] (its 128-row query tile holds G live rows: the MMA
        // has time to spare, and its pipeline streams K and V at the rate of HBM) when its
        // one CTA per SM covers the units in one wave or their key ranges are long; otherwise
        // (short contexts over more units than SMs: its per-CTA start would be paid twice)
        // the CUDA-core decode kernel, two CTAs per SM.  Measured on a GB300: Llama-3-8B
        // layer, 32 layers x 1 request, 1360 keys: 45 us CUDA cores, 52 us tensor cores;
        // 16 requests x 1160 keys: 31 / 28 us; 2 x 2300 keys, G = 8: 26 / 19 us; 8 x 32900
        // keys: 212 / 192 us.
        const int64_t tiles_max = (n_keys_max + 127) / 128;
        const bool use_tc = c->cfg.attn_impl != C2KV_ATTN_SIMT &&
                            c2kv::attn_tc_supported(c->cfg.dtype, d, hq, hkv) &&
                            (c->cfg.attn_impl == C2KV_ATTN_TC || units <= c->sms || tiles_max >= 32);
        int32_t n_split = 1;
        if (use_tc) {
            // splits per (layer, request, KV head): the fewest waves of one-CTA-per-SM work,
            // each CTA paying about four key tiles' time to start and finish, a split another
            // two for the merge
            const int64_t tiles = tiles_max;
            if (c->cfg.attn_split >= 1) {
                n_split = (int32_t)std::min<int64_t>(c->cfg.attn_split, tiles);
            } else {
                double best = 0.0;
                for (int32_t n = 1; n <= c2kv::kMaxMergeSplits && n <= tiles; ++n) {
                    const int64_t waves = (units * n + c->sms - 1) / c->sms;
                    const double t = (double)waves * ((double)((tiles + n - 1) / n) + 4.0) + (n > 1 ? 2.0 : 0.0);
                    if (n == 1 || t < best) {
                        best = t;
                        n_split = n;
                    }
                }
            }
        } else {
            // Key-range splits per (layer, request, KV head), from a model of the schedule: the
            // CTAs run in waves of (resident CTAs per SM) x SMs; a CTA spends a start latency
            // (about 2 us: its first tiles in flight) plus its keys' K/V bytes at its share of
            // HBM, at most what one CTA's consumer warps keep up with (about 25 GB/s,
            // measured); a split adds the merge (about 3 us).  Splits keep at least 128 keys.
            const int32_t grp = hq / hkv;
            const int64_t slots = (int64_t)(grp >= 8 ? 1 : 2) * c->sms;
            const double bytes_per_key = 2.0 * d * (double)c->eb;
            double best = 0.0;
            for (int32_t n = 1; n <= 64; ++n) {
                const int32_t kps = (n_keys_max + n - 1) / n;
                if (n > 1 && kps < 128) break;
                const int64_t ctas = units * n;
                const int64_t waves = (ctas + slots - 1) / slots;
                const double bw = std::min(6.0e12 / (double)std::min(ctas, slots), 25.0e9);
                const double t = (double)waves * (2e-6 + kps * bytes_per_key / bw) + (n > 1 ? 3e-6 : 0.0);
                if (n == 1 || t < best) {
                    best = t;
                    n_split = n;
                }
            }
        }
        const int32_t keys_per_split = (n_keys_max + n_split - 1) / n_split;

        const size_t q_bytes = (size_t)lq * B * hq * d * c->eb;
        void* q_rot = nullptr;
        cudaError_t e = pool_alloc(c, &q_rot, q_bytes);
        if (e != cudaSuccess) return cuda_fail(c, e, "decode: scratch allocation");
        float* part = nullptr;
        const size_t rows_all = (size_t)lq * B * hq;
        if (n_split > 1) {
            e = pool_alloc(c, reinterpret_cast<void**>(&part), (size_t)n_split * rows_all * (d + 1) * sizeof(float));
            // the tensor-core kernel merges the splits itself (per-unit counters)
            if (e == cudaSuccess && use_tc && n_split <= c2kv::kMaxMergeSplits)
                e = tickets_ready(c, (size_t)c2kv::attn_tc_units(hq, hkv, 1, lq, std::min<int32_t>(B, c2kv::kMaxReq)));
            if (e != cudaSuccess) {
                pool_free(c, part);
                pool_free(c, q_rot);
                return cuda_fail(c, e, "decode: split scratch allocation");
            }
        }
        // the tensor-core route reads whole 128-row key tiles: the rows after the new one up to
        // the next 128-row edge must hold finite values (masked keys weigh zero, but 0 * NaN is
        // not zero), so each request's are zeroed once, when not written or zeroed before
        std::vector<int32_t> edge(B), pad_from(B);
        bool any_pad = false;
        for (int32_t b = 0; b < B; ++b) {
            const int64_t next = (int64_t)cache->n_slots[b] + steps[b] + 1;
            edge[b] = (int32_t)std::min<int64_t>((next + kTileRows - 1) / kTileRows * kTileRows, cache->capacity[b]);
            bool need = false;
            for (int32_t l = layer0; use_tc && l < layer0 + lq; ++l)
                need = need || cache->clean_to[(size_t)l * B + b] < edge[b];
            pad_from[b] = need ? (int32_t)next : (int32_t)((next + kTileRows - 1) / kTileRows * kTileRows);
            any_pad = any_pad || need;
        }
        std::vector<c2kv::ReqParam> reqs(B);
        for (int32_t b = 0; b < B; ++b)
            reqs[b] = c2kv::ReqParam{cache->row_base[b], cache->n_slots[b], cache->l_req[b], steps[b]};
        for (int32_t b0 = 0; e == cudaSuccess && b0 < B; b0 += c2kv::kMaxReq) {
            const int32_t nb = std::min<int32_t>(c2kv::kMaxReq, B - b0);
            c2kv::SuffixParams s{};
            s.q = q;
            s.k = k_new;
            s.v = v_new;
            s.q_rot = q_rot;
            s.cache_k = cache->k;
            s.cache_v = cache->v;
            s.pos = cache->pos;
            s.rows = cache->rows;
            s.layer0 = layer0;
            s.lq = lq;
            s.batch = nb;
            s.batch_total = B;
            s.b0 = b0;
            s.sq = 1;
            s.hq = hq;
            s.hkv = hkv;
            s.pad_rows = any_pad ? 1 : 0;
            s.rope = c->turns;
            for (int32_t i = 0; i < nb; ++i) {
                s.req[i] = reqs[b0 + i];
                s.pad_from[i] = pad_from[b0 + i];
            }
            {
                ProfScope prof_suffix(c, C2KV_PROF_SUFFIX);
                e = c2kv::launch_suffix_prep(s, c->cfg.dtype, d, c->stream);
            }
            if (e != cudaSuccess) break;
            if (use_tc) {
                c2kv::AttnParams a{};
                a.q_rot = q_rot;
                a.cache_k = cache->k;
                a.cache_v = cache->v;
                a.out = out;
                a.lse = lse;
                a.err = c->d_err;
                a.rows = cache->rows;
                a.layer0 = layer0;
                a.lq = lq;
                a.batch = nb;
                a.batch_total = B;
                a.b0 = b0;
                a.sq = 1;
                a.hq = hq;
                a.hkv = hkv;
                a.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)d));
                a.n_split = n_split;
                a.pairs_per_cta = c->cfg.attn_pairs;
                a.part_o = part;
                a.part_lse = part ? part + (size_t)n_split * rows_all * d : nullptr;
                // the splits merged in the kernel (beyond kMaxMergeSplits: by a launch after the
                // last group)
                const bool in_kernel = n_split > 1 && n_split <= c2kv::kMaxMergeSplits;
                a.tickets = in_kernel ? c->tickets : nullptr;
                // the two softmax warpgroups take alternate key tiles of the one query tile
                a.key_pingpong = 1;
                // the suffix kernel's programmatic dependent, unless a trace puts events
                // between them
                a.dependent = c->prof ? 0 : 1;
                for (int32_t i = 0; i < nb; ++i) a.req[i] = reqs[b0 + i];
                ProfScope prof_decode(c, C2KV_PROF_DECODE, true);
                e = c2kv::launch_attn_tc(a, c->stream, prof_decode.hook());
                if (e == cudaSuccess && n_split > 1 && !in_kernel && b0 + nb >= B)
                    e = c2kv::launch_attn_combine(a, c->stream);
                continue;
            }
            c2kv::DecodeParams p{};
            p.q_rot = q_rot;
            p.cache_k = cache->k;
            p.cache_v = cache->v;
            p.out = out;
            p.lse = lse;
            p.part_o = part;
            p.part_lse = part ? part + (size_t)n_split * rows_all * d : nullptr;
            p.err = c->d_err;
            p.rows = cache->rows;
            p.layer0 = layer0;
            p.lq = lq;
            p.batch = nb;
            p.batch_total = B;
            p.b0 = b0;
            p.hq = hq;
            p.hkv = hkv;
            p.d = d;
            p.n_split = n_split;
            p.keys_per_split = keys_per_split;
            p.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)d));
            p.dependent = c->prof ? 0 : 1;    // a trace records events between the two kernels
            for (int32_t i = 0; i < nb; ++i) p.req[i] = s.req[i];
            ProfScope prof_decode(c, C2KV_PROF_DECODE, true);
            e = c2kv::launch_decode(p, c->cfg.dtype, c->stream, prof_decode.hook());
        }
        pool_free(c, part);
        pool_free(c, q_rot);
        if (e != cudaSuccess) return cuda_fail(c, e, "decode");
        for (int32_t l = layer0; l < layer0 + lq; ++l)
            for (int32_t b = 0; b < B; ++b) {
                int32_t& ct = cache->clean_to[(size_t)l * B + b];
                ct = std::max(ct, pad_from[b] < edge[b] ? edge[b] : cache->n_slots[b] + steps[b] + 1);
            }
        return C2KV_OK;
    } catch (const std::bad_alloc&) {
        return fail(c, C2KV_ERR_NOMEM, "decode: host allocation failed");
    }
}

c2kv_status c2kv_extract_attention(c2kv_ctx* c, int32_t n_layers, const void* q, const void* k,
                                   const void* v, int32_t n_tokens, int32_t ratio_k, void* out,
                                   float* lse) {
    if (!c) return C2KV_ERR_ARG;
    try {
        c->err.clear();
        if (!q || !k || !v || !out) return fail(c, C2KV_ERR_ARG, "extract: null pointer");
        if (!aligned(q) || !aligned(k) || !aligned(v) || !aligned(out) || !aligned(lse, 4))
            return fail(c, C2KV_ERR_ARG, "extract: misaligned tensor pointer");
        if (const c2kv_status st = require_device(c, "extract", {q, k, v, out, lse})) return st;
        if (n_layers < 1 || n_tokens < 1 || ratio_k < 1)
            return fail(c, C2KV_ERR_ARG, "extract: need n_layers, n_tokens, ratio_k >= 1");
        const int32_t d = c->cfg.head_dim;
        if (d != 64 && d != 128) return fail(c, C2KV_ERR_UNSUPPORTED, "extract: head_dim %d", d);
        const int64_t m = ((int64_t)n_tokens + ratio_k - 1) / ratio_k;
        if ((int64_t)n_tokens + m > 0x7fffffffLL / 128) return fail(c, C2KV_ERR_ARG, "extract: chunk too long");
        const int32_t n_all = (int32_t)(n_tokens + m);
        const int32_t hq = c->cfg.n_q_heads, hkv = c->cfg.n_kv_heads;
        const size_t qb = (size_t)n_layers * n_all * hq * d * c->eb;
        const size_t kb = (size_t)n_layers * n_all * hkv * d * c->eb;
        void* q_rot = nullptr;
        void* k_rot = nullptr;
        cudaError_t e = pool_alloc(c, &q_rot, qb);
        if (e == cudaSuccess) e = pool_alloc(c, &k_rot, kb);
        if (e != cudaSuccess) {
            if (k_rot) pool_free(c, k_rot);
            if (q_rot) pool_free(c, q_rot);
            return cuda_fail(c, e, "extract: scratch allocation");
        }
        c2kv::ExtractParams p{};
        p.err = c->d_err;
        p.q = q;
        p.k = k;
        p.v = v;
        p.q_rot = q_rot;
        p.k_rot = k_rot;
        p.out = out;
        p.lse = lse;
        p.lq = n_layers;
        p.n = n_tokens;
        p.ratio = ratio_k;
        p.n_all = n_all;
        p.hq = hq;
        p.hkv = hkv;
        p.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)d));
        p.pairs_per_cta = c->cfg.attn_pairs;
        p.rope = c->turns;
        // the C2 rows beside the document rows on the second stream (tensor-core route)
        const bool two = c2kv::extract_uses_tc(c->cfg.dtype, d, c->cfg.n_q_heads, c->cfg.n_kv_heads) &&
                         aux_ready(c, 2) == cudaSuccess;
        {
            ProfScope prof(c, C2KV_PROF_EXTRACT);
            e = c2kv::launch_extract(p, c->cfg.dtype, d, c->stream, two ? c->aux : nullptr,
                                     two ? c->aux_ev[0] : nullptr, two ? c->aux_ev[1] : nullptr);
        }
        if (e != cudaSuccess && two) cudaStreamSynchronize(c->aux);   // before the scratch goes
        pool_free(c, k_rot);
        pool_free(c, q_rot);
        if (e != cudaSuccess) return cuda_fail(c, e, "extract");
        return C2KV_OK;
    } catch (const std::bad_alloc&) {
        return fail(c, C2KV_ERR_NOMEM, "extract: host allocation failed");
    }
}

c2kv_status c2kv_cache_release(c2kv_ctx* c, c2kv_cache* cache) {
    if (!c) return C2KV_ERR_ARG;
    c->err.clear();
    if (!own_cache(c, cache)) return fail(c, C2KV_ERR_STATE, "cache_release: cache not owned by this context");
    c->caches.erase(std::find(c->caches.begin(), c->caches.end(), cache));
    destroy_cache(c, cache);
    return C2KV_OK;
}

c2kv_status c2kv_sync(c2kv_ctx* c) {
    if (!c) return C2KV_ERR_ARG;
    c->err.clear();
    cudaError_t e = cudaStreamSynchronize(c->stream);
    if (e != cudaSuccess) return cuda_fail(c, e, "sync");
    int32_t word = 0;
    e = cudaMemcpy(&word, c->d_err, sizeof(word), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(c, e, "sync: error word");
    if (word != 0) {
        cudaMemset(c->d_err, 0, sizeof(int32_t));
        // a launch that gave up may have left split-merge counters part-way
        if (c->tickets) cudaMemsetAsync(c->tickets, 0, c->tickets_cap * sizeof(uint32_t), c->stream);
        return fail(c, C2KV_ERR_DEVICE_BOUNDS, "sync: a kernel refused an out-of-range index (flags 0x%x)", word);
    }
    return C2KV_OK;
}

c2kv_status c2kv_profile_enable(c2kv_ctx* c, int32_t on) {
    if (!c) return C2KV_ERR_ARG;
    c->prof = on != 0;
    // create the trace's events now, so that a traced call only records them: creating
    // events inside the calls would slow the host enough to delay the launches it traces
    try {
        const size_t have = c->prof_free.size() + 2 * c->prof_recs.size();
        for (size_t i = have; c->prof && i < kProfEvents; ++i) {
            cudaEvent_t e = nullptr;
            if (cudaEventCreate(&e) != cudaSuccess) {
                (void)cudaGetLastError();
                break;
            }
            c->prof_free.push_back(e);
        }
    } catch (const std::bad_alloc&) {
    }
    return C2KV_OK;
}

c2kv_status c2kv_profile_read(c2kv_ctx* c, float* mean_ms, int32_t* launches) {
    if (!c) return C2KV_ERR_ARG;
    try {
        c->err.clear();
        cudaError_t e = cudaStreamSynchronize(c->stream);
        if (e != cudaSuccess) return cuda_fail(c, e, "profile_read");
        double sum[C2KV_PROF_KINDS] = {0};
        int32_t cnt[C2KV_PROF_KINDS] = {0};
        for (auto& r : c->prof_recs) {
            float ms = 0.f;
            if (cudaEventElapsedTime(&ms, r.a, r.b) == cudaSuccess && r.kind >= 0 &&
                r.kind < C2KV_PROF_KINDS) {
                sum[r.kind] += ms;
                cnt[r.kind] += 1;
            }
            (void)cudaGetLastError();
            c->prof_free.push_back(r.a);
            c->prof_free.push_back(r.b);
        }
        c->prof_recs.clear();
        for (int k = 0; k < C2KV_PROF_KINDS; ++k) {
            if (mean_ms) mean_ms[k] = cnt[k] ? (float)(sum[k] / cnt[k]) : 0.f;
            if (launches) launches[k] = cnt[k];
        }
        return C2KV_OK;
    } catch (const std::bad_alloc&) {
        return fail(c, C2KV_ERR_NOMEM, "profile_read: host allocation failed");
    }
}

c2kv_status c2kv_inject_fault(c2kv_ctx* c, int32_t what) {
    if (!c) return C2KV_ERR_ARG;
    if (what < 0 || what > 1) return fail(c, C2KV_ERR_ARG, "inject_fault: unknown fault %d", what);
    c->inject = what;
    return C2KV_OK;
}

}  // extern "C"

namespace c2kv {

bool attend_view(const c2kv_ctx* c, const c2kv_cache* cache, AttendView* v) {
    if (!c || !v || !own_cache(c, cache)) return false;
    v->layers = c->cfg.layers;
    v->n_q_heads = c->cfg.n_q_heads;
    v->n_kv_heads = c->cfg.n_kv_heads;
    v->head_dim = c->cfg.head_dim;
    v->dtype = c->cfg.dtype;
    v->attn_impl = c->cfg.attn_impl;
    v->attn_pairs = c->cfg.attn_pairs;
    v->device = c->device;
    v->noalloc_scratch = c->noalloc_scratch;
    v->stream = c->stream;
    v->err = c->d_err;
    v->turns = c->turns;
    v->cache_k = cache->k;
    v->cache_v = cache->v;
    v->pos = cache->pos;
    v->rows = cache->rows;
    v->batch = cache->batch;
    v->suffix_capacity = cache->suffix_capacity;
    v->row_base = cache->row_base.data();
    v->n_slots = cache->n_slots.data();
    v->l_req = cache->l_req.data();
    return true;
}

void note_suffix_written(c2kv_cache* cache, int32_t l0, int32_t n, int32_t n_suffix) {
    mark_suffix_clean(cache, l0, n, n_suffix);
}

MemKind mem_kind(const void* p) {
    if (!p) return MemKind::kDevice;
    cudaPointerAttributes a{};
    if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
        (void)cudaGetLastError();
        return MemKind::kUnknown;
    }
    if (a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged) return MemKind::kDevice;
    if (a.type == cudaMemoryTypeHost && a.devicePointer == p) return MemKind::kHost;
    return MemKind::kUnknown;
}

int32_t set_last_error(c2kv_ctx* c, int32_t code, const char* msg) {
    if (c) c->err = msg ? msg : "";
    return code;
}

}  // namespace c2kv
