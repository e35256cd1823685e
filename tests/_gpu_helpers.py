"""Shared helpers for the GPU parity tests: build inputs from synth, run the C ABI, run the
oracle on the same inputs, and compare with the tolerances the tests state."""
from __future__ import annotations

import numpy as np
import torch

import synth
from oracle import c2kv_oracle as orc

ATTN_TOL = {"bf16": 2e-2, "f32": 1e-5}


def lib():
    import __graft_entry__ as g
    g.build()
    from paper_2607_17715_gb300 import c2kv
    return c2kv


def tdtype(wl):
    return torch.float32 if wl.dtype == "f32" else torch.bfloat16


def dcode(wl):
    c2kv = lib()
    return c2kv.DTYPE_F32 if wl.dtype == "f32" else c2kv.DTYPE_BF16


def to_dev(x, wl):
    return torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).to("cuda", tdtype(wl))


def make_ctx(wl, pool_slots, attn_impl=0, fixed_pos=0, attn_split=0, fuse=0, storage=0, attn_pairs=0):
    c2kv = lib()
    return c2kv.c2kv_create(wl.layers, wl.n_q_heads, wl.n_kv_heads, wl.head_dim, wl.rope_theta,
                            dcode(wl), pool_slots, fixed_pos=fixed_pos, attn_impl=attn_impl,
                            stream=torch.cuda.current_stream(), attn_split=attn_split, fuse=fuse,
                            storage=storage, attn_pairs=attn_pairs)


def pool_rows(ctx, wl, chunk_id, pool_slots):
    """Read a chunk's stored slots back from the device pool: (K, V) [L, m, Hkv, d] fp64."""
    c2kv = lib()
    info = c2kv.c2kv_chunk_info(ctx, chunk_id)
    m = info["n_slots"]
    out = []
    for key in ("k", "v"):
        ptr = info[key] - info["slot_base"] * wl.n_kv_heads * wl.head_dim * (
            4 if wl.dtype == "f32" else 2)
        full = c2kv.device_view(ptr, (wl.layers, pool_slots, wl.n_kv_heads, wl.head_dim),
                                tdtype(wl))
        sl = full[:, info["slot_base"]:info["slot_base"] + m]
        out.append(sl.double().cpu().numpy())
    return out[0], out[1]


def cache_arrays(cache, wl):
    """(info, K, V, pos) of a composed cache: K/V [L, rows, Hkv, d] fp64, pos [rows] int."""
    c2kv = lib()
    info = c2kv.c2kv_cache_info(cache)
    shp = (info["layers"], info["rows"], wl.n_kv_heads, wl.head_dim)
    k = c2kv.device_view(info["k"], shp, tdtype(wl)).double().cpu().numpy()
    v = c2kv.device_view(info["v"], shp, tdtype(wl)).double().cpu().numpy()
    pos = c2kv.device_view(info["pos"], (info["rows"],), torch.int32).cpu().numpy()
    return info, k, v, pos


def order_keys(x: np.ndarray, wl) -> np.ndarray:
    """Monotone integer keys of the storage encoding (adjacent representable values differ
    by 1), so key differences count ulps."""
    if wl.dtype == "bf16":
        b = torch.from_numpy(np.asarray(x, np.float32)).to(torch.bfloat16).view(torch.int16)
        b = b.numpy().astype(np.int64)
        return np.where(b < 0, -(b & 0x7FFF), b)
    b = np.asarray(x, np.float32).view(np.int32).astype(np.int64)
    return np.where(b < 0, -(b & 0x7FFFFFFF), b)


def ulp_of(x: np.ndarray, wl) -> np.ndarray:
    bits = 8 if wl.dtype == "bf16" else 24
    x = np.abs(np.asarray(x, np.float64))
    e = np.frexp(np.where(x == 0, 1e-38, x))[1]
    return np.exp2(e - bits)


def pair_magnitude(k_stored: np.ndarray) -> np.ndarray:
    """|(x_i, x_{i+d/2})| for every channel of every row (rotation keeps it fixed)."""
    d = k_stored.shape[-1]
    a, b = k_stored[..., : d // 2], k_stored[..., d // 2:]
    m = np.sqrt(a * a + b * b)
    return np.concatenate([m, m], axis=-1)


def check_rounded(got, want, scale, wl, what):
    """At most one storage ulp from the fp64 result rounded once, or within fp32
    arithmetic error, 2^-20 of `scale` (the magnitude of the operands the value was
    computed from), where the result is much smaller than its operands."""
    diff = np.abs(got - want)
    allowed = np.maximum(ulp_of(want, wl), 2.0 ** -20 * scale)
    bad = diff > allowed
    assert not bad.any(), (f"{what}: {bad.sum()} elements off; worst diff "
                           f"{diff.max():.3g}, ulps {np.max(np.abs(order_keys(got, wl) - order_keys(want, wl)))}")


def check_rotated(got, want, k_stored, wl, what):
    """Rotated K: at most one storage ulp from the fp64 result rounded once, or within the
    fp32 arithmetic error of the rotation (2^-20 of the pair's magnitude) where a pair
    nearly cancels."""
    diff = np.abs(got - want)
    allowed = np.maximum(ulp_of(want, wl), 2.0 ** -20 * pair_magnitude(k_stored))
    bad = diff > allowed
    assert not bad.any(), (f"{what}: {bad.sum()} elements off; worst diff "
                           f"{diff.max():.3g}, ulps {np.max(np.abs(order_keys(got, wl) - order_keys(want, wl)))}")


def check_attention(got, want, wl, what):
    tol = ATTN_TOL[wl.dtype]
    diff = np.abs(got - want)
    bad = diff > tol + tol * np.abs(want)
    assert np.isfinite(got).all(), f"{what}: non-finite output"
    assert not bad.any(), (f"{what}: {bad.sum()} of {bad.size} outside atol=rtol={tol}; "
                           f"max abs {diff.max():.3g}")


def oracle_chunks_meanpool(wl, ids):
    """Oracle-compressed chunks (stored form) for the given pool ids."""
    out = {}
    for cid in ids:
        kt, vt = synth.chunk_tokens(wl, cid)
        ks, vs = orc.compress_chunk(kt, vt, wl.chunk_tokens, wl.ratio_k, wl.rope_theta,
                                    wl.dtype, "meanpool")
        out[cid] = (ks, vs, wl.chunk_tokens, wl.ratio_k)
    return out


def load_stored(ctx, wl, chunks, host=(), keep=None):
    """Register stored-form chunks: copied into the device pool (MODE_STORED), or, for the
    ids in `host`, left in pinned host memory (MODE_HOST; the pinned tensors are appended to
    `keep`, which must outlive the chunks).  Returns the library id of every chunk."""
    c2kv = lib()
    ids = {}
    for cid, (ks, vs, n, k) in chunks.items():
        if cid in host:
            kh, vh = (torch.from_numpy(np.ascontiguousarray(x, np.float32)).to(tdtype(wl))
                      .pin_memory() for x in (ks, vs))
            keep.extend((kh, vh))
            ids[cid] = c2kv.c2kv_compress_chunk(ctx, kh, vh, n, k, c2kv.MODE_HOST)
        else:
            ids[cid] = c2kv.c2kv_compress_chunk(ctx, to_dev(ks, wl), to_dev(vs, wl), n, k,
                                                c2kv.MODE_STORED)
    return ids
