"""Thin Python binding of libc2kv (the C ABI in include/c2kv.h).

Argument marshalling only: every function here has the name of the C entry point it
calls, turns torch tensors / numpy arrays into raw pointers, and raises ``C2KVError``
on a non-OK status.  No computation of the method happens in Python, and there is no
fallback: if the compiled library is missing, importing this module fails.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_lib", "libc2kv.so")

if not os.path.exists(LIB_PATH):
    raise ImportError(
        f"libc2kv.so not found at {LIB_PATH}: build it first "
        "(python -c 'import __graft_entry__ as g; g.build()')")

_lib = ctypes.CDLL(LIB_PATH)

# status codes / enums (mirror include/c2kv.h)
OK = 0
ERR_ARG, ERR_DTYPE, ERR_NOMEM, ERR_POOL_FULL, ERR_BAD_CHUNK = -1, -2, -3, -4, -5
ERR_POSITIONS, ERR_CUDA, ERR_DEVICE_BOUNDS, ERR_STATE, ERR_UNSUPPORTED = -6, -7, -8, -9, -10
DTYPE_BF16, DTYPE_F32 = 0, 1
MODE_MEANPOOL, MODE_PROVIDED, MODE_STORED, MODE_HOST = 0, 1, 2, 3
ATTN_AUTO, ATTN_SIMT, ATTN_TC = 0, 1, 2
FUSE_AUTO, FUSE_NEVER, FUSE_ALWAYS = 0, 1, 2
STORAGE_LOCAL_ROPE, STORAGE_PRE_ROPE = 0, 1
PROF_COMPOSE, PROF_COMPRESS, PROF_SUFFIX, PROF_ATTN, PROF_COMBINE, PROF_DECODE = 0, 1, 2, 3, 4, 5
PROF_EXTRACT, PROF_FUSED = 6, 7
PROF_KINDS = 8
PROF_NAMES = ("compose", "compress", "suffix", "attention", "combine", "decode", "extract",
              "fused")

STATUS_NAMES = {
    0: "OK", -1: "ERR_ARG", -2: "ERR_DTYPE", -3: "ERR_NOMEM", -4: "ERR_POOL_FULL",
    -5: "ERR_BAD_CHUNK", -6: "ERR_POSITIONS", -7: "ERR_CUDA", -8: "ERR_DEVICE_BOUNDS",
    -9: "ERR_STATE", -10: "ERR_UNSUPPORTED",
}


class c2kv_config(ctypes.Structure):
    _fields_ = [("layers", ctypes.c_int32), ("n_q_heads", ctypes.c_int32),
                ("n_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("rope_theta", ctypes.c_double), ("dtype", ctypes.c_int32),
                ("pool_slots", ctypes.c_int32), ("fixed_pos", ctypes.c_int32),
                ("attn_impl", ctypes.c_int32), ("attn_split", ctypes.c_int32),
                ("fuse", ctypes.c_int32), ("storage", ctypes.c_int32),
                ("attn_pairs", ctypes.c_int32)]


class c2kv_chunk_desc(ctypes.Structure):
    _fields_ = [("n_tokens", ctypes.c_int32), ("ratio_k", ctypes.c_int32),
                ("n_slots", ctypes.c_int32), ("slot_base", ctypes.c_int32),
                ("k", ctypes.c_void_p), ("v", ctypes.c_void_p),
                ("layer_stride", ctypes.c_int64)]


_P32 = ctypes.POINTER(ctypes.c_int32)


class c2kv_cache_desc(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("layers", ctypes.c_int32),
                ("rows", ctypes.c_int64), ("k", ctypes.c_void_p), ("v", ctypes.c_void_p),
                ("pos", ctypes.c_void_p), ("row_base", _P32), ("n_slots", _P32),
                ("l_req", _P32), ("capacity", _P32), ("suffix_capacity", ctypes.c_int32)]


_VP, _I32 = ctypes.c_void_p, ctypes.c_int32
_SIGS = {
    "c2kv_abi_version": (_I32, []),
    "c2kv_create": (_I32, [ctypes.POINTER(c2kv_config), _VP, ctypes.POINTER(_VP)]),
    "c2kv_destroy": (_I32, [_VP]),
    "c2kv_set_stream": (_I32, [_VP, _VP]),
    "c2kv_compress_chunk": (_I32, [_VP, _VP, _VP, _I32, _I32, _I32, _P32]),
    "c2kv_free_chunk": (_I32, [_VP, _I32]),
    "c2kv_chunk_info": (_I32, [_VP, _I32, ctypes.POINTER(c2kv_chunk_desc)]),
    "c2kv_compose": (_I32, [_VP, _I32, _P32, _P32, _P32, _I32, ctypes.POINTER(_VP)]),
    "c2kv_compose_attend": (_I32, [_VP, _I32, _P32, _P32, _P32, _I32, _VP, _VP, _VP, _I32, _VP,
                                   _VP, ctypes.POINTER(_VP)]),
    "c2kv_cache_info": (_I32, [_VP, ctypes.POINTER(c2kv_cache_desc)]),
    "c2kv_attend": (_I32, [_VP, _VP, _I32, _VP, _VP, _VP, _I32, _VP, _VP]),
    "c2kv_attend_noalloc": (_I32, [_VP, _VP, _I32, _VP, _VP, _VP, _I32, _VP, _VP]),
    "c2kv_decode": (_I32, [_VP, _VP, _I32, _VP, _VP, _VP, _P32, _VP, _VP]),
    "c2kv_extract_attention": (_I32, [_VP, _I32, _VP, _VP, _VP, _I32, _I32, _VP, _VP]),
    "c2kv_cache_release": (_I32, [_VP, _VP]),
    "c2kv_sync": (_I32, [_VP]),
    "c2kv_last_error": (ctypes.c_char_p, [_VP]),
    "c2kv_inject_fault": (_I32, [_VP, _I32]),
    "c2kv_profile_enable": (_I32, [_VP, _I32]),
    "c2kv_profile_read": (_I32, [_VP, ctypes.POINTER(ctypes.c_float), _P32]),
}
for _name, (_res, _args) in _SIGS.items():
    _fn = getattr(_lib, _name)
    _fn.restype = _res
    _fn.argtypes = _args


class C2KVError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {message}")
        self.status = status


def _check(status: int, ctx=None):
    if status != OK:
        raise C2KVError(status, c2kv_last_error(ctx))


def _ptr(x):
    """Raw address of a torch tensor, numpy array, int or None."""
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if hasattr(x, "data_ptr"):
        return x.data_ptr()
    if isinstance(x, np.ndarray):
        return x.ctypes.data
    raise TypeError(f"cannot take the address of {type(x)}")


def _i32(arr):
    if arr is None:
        return None, None
    a = np.ascontiguousarray(np.asarray(arr, dtype=np.int32))
    return a, a.ctypes.data_as(_P32)


def _stream_handle(stream):
    if stream is None:
        return None
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


# ---------------------------------------------------------------------------- calls

def c2kv_abi_version() -> int:
    return _lib.c2kv_abi_version()


def c2kv_last_error(ctx=None) -> str:
    msg = _lib.c2kv_last_error(ctx)
    return msg.decode() if msg else ""


def c2kv_create(layers, n_q_heads, n_kv_heads, head_dim, rope_theta, dtype, pool_slots,
                fixed_pos=0, attn_impl=ATTN_AUTO, stream=None, attn_split=0, fuse=0,
                storage=STORAGE_LOCAL_ROPE, attn_pairs=0):
    cfg = c2kv_config(layers, n_q_heads, n_kv_heads, head_dim, float(rope_theta), dtype,
                      pool_slots, int(fixed_pos), attn_impl, attn_split, fuse, storage, attn_pairs)
    out = _VP()
    _check(_lib.c2kv_create(ctypes.byref(cfg), _stream_handle(stream), ctypes.byref(out)))
    return out.value


def c2kv_destroy(ctx):
    _check(_lib.c2kv_destroy(ctx), None)


def c2kv_set_stream(ctx, stream):
    _check(_lib.c2kv_set_stream(ctx, _stream_handle(stream)), ctx)


def c2kv_compress_chunk(ctx, k, v, n_tokens, ratio_k, mode) -> int:
    cid = ctypes.c_int32(-1)
    _check(_lib.c2kv_compress_chunk(ctx, _ptr(k), _ptr(v), n_tokens, ratio_k, mode,
                                    ctypes.byref(cid)), ctx)
    return cid.value


def c2kv_free_chunk(ctx, chunk_id):
    _check(_lib.c2kv_free_chunk(ctx, chunk_id), ctx)


def c2kv_chunk_info(ctx, chunk_id) -> dict:
    d = c2kv_chunk_desc()
    _check(_lib.c2kv_chunk_info(ctx, chunk_id, ctypes.byref(d)), ctx)
    return {f: getattr(d, f) for f, _ in c2kv_chunk_desc._fields_}


def c2kv_compose(ctx, req_ptr, chunk_ids, positions=None, suffix_capacity=0):
    rp, rp_p = _i32(req_ptr)
    ids, ids_p = _i32(chunk_ids)
    pos, pos_p = _i32(positions)
    out = _VP()
    _check(_lib.c2kv_compose(ctx, len(rp) - 1, rp_p, ids_p, pos_p, suffix_capacity,
                             ctypes.byref(out)), ctx)
    return out.value


def c2kv_compose_attend(ctx, req_ptr, chunk_ids, positions, suffix_capacity, q, k_suf, v_suf,
                        n_suffix, out, lse=None):
    """Compose the requests' chunks and attend their suffixes over all layers in one call
    (fused on the tensor-core route); returns the composed cache."""
    rp, rp_p = _i32(req_ptr)
    ids, ids_p = _i32(chunk_ids)
    pos, pos_p = _i32(positions)
    cache = _VP()
    _check(_lib.c2kv_compose_attend(ctx, len(rp) - 1, rp_p, ids_p, pos_p, suffix_capacity, _ptr(q),
                                    _ptr(k_suf), _ptr(v_suf), n_suffix, _ptr(out), _ptr(lse),
                                    ctypes.byref(cache)), ctx)
    return cache.value


def c2kv_cache_info(cache) -> dict:
    d = c2kv_cache_desc()
    _check(_lib.c2kv_cache_info(cache, ctypes.byref(d)))
    b = d.batch
    return dict(batch=b, layers=d.layers, rows=d.rows, k=d.k, v=d.v, pos=d.pos,
                row_base=np.ctypeslib.as_array(d.row_base, (b,)).copy(),
                n_slots=np.ctypeslib.as_array(d.n_slots, (b,)).copy(),
                l_req=np.ctypeslib.as_array(d.l_req, (b,)).copy(),
                capacity=np.ctypeslib.as_array(d.capacity, (b,)).copy(),
                suffix_capacity=d.suffix_capacity)


def c2kv_attend(ctx, cache, layer, q, k_suf, v_suf, n_suffix, out, lse=None):
    _check(_lib.c2kv_attend(ctx, cache, layer, _ptr(q), _ptr(k_suf), _ptr(v_suf), n_suffix,
                            _ptr(out), _ptr(lse)), ctx)


def c2kv_attend_noalloc(ctx, cache, layer, q, k_suf, v_suf, n_suffix, out, lse=None):
    """c2kv_attend without any device allocation (scratch in a fixed 16 MiB device array;
    see include/c2kv.h for the limits)."""
    _check(_lib.c2kv_attend_noalloc(ctx, cache, layer, _ptr(q), _ptr(k_suf), _ptr(v_suf),
                                    n_suffix, _ptr(out), _ptr(lse)), ctx)


def c2kv_decode(ctx, cache, layer, q, k_new, v_new, steps, out, lse=None):
    """One decode step: request r's new token at suffix index steps[r] (host int array)."""
    st, st_p = _i32(steps)
    _check(_lib.c2kv_decode(ctx, cache, layer, _ptr(q), _ptr(k_new), _ptr(v_new), st_p,
                            _ptr(out), _ptr(lse)), ctx)


def c2kv_extract_attention(ctx, n_layers, q, k, v, n_tokens, ratio_k, out, lse=None):
    """SIF-masked extraction attention over [document tokens; C2 tokens] of one chunk."""
    _check(_lib.c2kv_extract_attention(ctx, n_layers, _ptr(q), _ptr(k), _ptr(v), n_tokens,
                                       ratio_k, _ptr(out), _ptr(lse)), ctx)


def c2kv_cache_release(ctx, cache):
    _check(_lib.c2kv_cache_release(ctx, cache), ctx)


def c2kv_sync(ctx):
    _check(_lib.c2kv_sync(ctx), ctx)


def c2kv_profile_enable(ctx, on=True):
    _check(_lib.c2kv_profile_enable(ctx, int(bool(on))), ctx)


def c2kv_profile_read(ctx) -> dict:
    """{kind name: (mean ms, launches)} for the launches recorded since the last read."""
    ms = (ctypes.c_float * PROF_KINDS)()
    cnt = (ctypes.c_int32 * PROF_KINDS)()
    _check(_lib.c2kv_profile_read(ctx, ms, cnt), ctx)
    return {PROF_NAMES[k]: (ms[k], cnt[k]) for k in range(PROF_KINDS)}


def c2kv_inject_fault(ctx, what):
    _check(_lib.c2kv_inject_fault(ctx, what), ctx)


# ---------------------------------------------------------------- device memory views

class _CudaArray:
    """Minimal __cuda_array_interface__ wrapper so torch can view library-owned memory."""

    def __init__(self, ptr, shape, typestr):
        self.__cuda_array_interface__ = {
            "shape": tuple(int(s) for s in shape), "typestr": typestr,
            "data": (int(ptr), False), "version": 2, "strides": None,
        }


def device_view(ptr, shape, dtype):
    """A torch tensor aliasing library-owned device memory (no copy).  Valid only while
    the owning object (cache, pool) lives."""
    import torch
    if dtype == torch.bfloat16:
        t = torch.as_tensor(_CudaArray(ptr, shape, "<i2"), device="cuda")
        return t.view(torch.bfloat16)
    typestr = {torch.float32: "<f4", torch.int32: "<i4"}[dtype]
    return torch.as_tensor(_CudaArray(ptr, shape, typestr), device="cuda")
