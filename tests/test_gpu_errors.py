"""Error paths of the C ABI on a live context: every refused call returns its status,
leaves state unchanged, and the context keeps working.  The device-side bounds check is
exercised by host-side fault injection (a corrupted slot map that the compose kernel
refuses and skips); nothing here faults the GPU."""
import numpy as np
import pytest
import torch

import synth
from tests import _gpu_helpers as H

pytestmark = pytest.mark.gpu

WL = synth.scaled(synth.workload("llama8b"), layers=2, chunk_tokens=64, ratio_k=4)


@pytest.fixture
def ctx():
    c2kv = H.lib()
    c = H.make_ctx(WL, pool_slots=64)
    yield c
    c2kv.c2kv_destroy(c)


def _chunk(ctx, cid=0, n=64, k=4):
    c2kv = H.lib()
    kt, vt = synth.chunk_tokens(WL, cid, n_tokens=n)
    return c2kv.c2kv_compress_chunk(ctx, H.to_dev(kt, WL), H.to_dev(vt, WL), n, k,
                                    c2kv.MODE_MEANPOOL)


def _status(fn, *a, **kw):
    c2kv = H.lib()
    try:
        fn(*a, **kw)
    except c2kv.C2KVError as e:
        return e.status
    return c2kv.OK


def test_bad_create_args():
    c2kv = H.lib()
    assert _status(c2kv.c2kv_create, 1, 4, 3, 128, 1e4, 0, 16) == c2kv.ERR_ARG     # Hq % Hkv
    assert _status(c2kv.c2kv_create, 1, 4, 2, 128, 1e4, 7, 16) == c2kv.ERR_DTYPE
    assert _status(c2kv.c2kv_create, 1, 4, 2, 128, 1e4, 0, 0) == c2kv.ERR_ARG
    assert _status(c2kv.c2kv_create, 1, 4, 2, 128, 1e4, 0, 1 << 30) == c2kv.ERR_NOMEM


def test_pool_full_leaves_state(ctx):
    c2kv = H.lib()
    a = _chunk(ctx)                       # 16 slots
    b = _chunk(ctx, 1)                    # 16
    c = _chunk(ctx, 2)                    # 16
    assert _status(_chunk, ctx, 3, 128, 4) == c2kv.ERR_POOL_FULL     # needs 32, 16 free
    d = _chunk(ctx, 3)                    # the last 16 still fit
    c2kv.c2kv_free_chunk(ctx, b)
    c2kv.c2kv_free_chunk(ctx, c)          # frees merge into one 32-slot range
    e = _chunk(ctx, 4, 128, 4)
    assert c2kv.c2kv_chunk_info(ctx, e)["n_slots"] == 32
    for x in (a, d, e):
        assert c2kv.c2kv_chunk_info(ctx, x)["n_slots"] in (16, 32)
    c2kv.c2kv_sync(ctx)


def test_bad_chunk_and_positions(ctx):
    c2kv = H.lib()
    a = _chunk(ctx)
    assert _status(c2kv.c2kv_free_chunk, ctx, 99) == c2kv.ERR_BAD_CHUNK
    assert _status(c2kv.c2kv_compose, ctx, [0, 1], [a + 5], [0], 4) == c2kv.ERR_BAD_CHUNK
    assert _status(c2kv.c2kv_compose, ctx, [0, 2], [a, a], [0, 10], 4) == c2kv.ERR_POSITIONS
    assert _status(c2kv.c2kv_compose, ctx, [0, 2], [a, a], [100, 0], 4) == c2kv.ERR_POSITIONS
    assert _status(c2kv.c2kv_compose, ctx, [0, 1], [a], [-3], 4) == c2kv.ERR_POSITIONS
    assert _status(c2kv.c2kv_compose, ctx, [1, 1], [a], [0], 4) == c2kv.ERR_ARG
    assert _status(c2kv.c2kv_compose, ctx, [0, 2, 1], [a, a], [0, 64], 4) == c2kv.ERR_ARG
    c2kv.c2kv_free_chunk(ctx, a)
    assert _status(c2kv.c2kv_free_chunk, ctx, a) == c2kv.ERR_BAD_CHUNK
    assert _status(c2kv.c2kv_compose, ctx, [0, 1], [a], [0], 4) == c2kv.ERR_BAD_CHUNK
    assert "unknown chunk" in c2kv.c2kv_last_error(ctx)


def test_compress_arg_checks(ctx):
    c2kv = H.lib()
    kt, vt = synth.chunk_tokens(WL, 0, n_tokens=8)
    kd, vd = H.to_dev(kt, WL), H.to_dev(vt, WL)
    assert _status(c2kv.c2kv_compress_chunk, ctx, kd, vd, 0, 4, 0) == c2kv.ERR_ARG
    assert _status(c2kv.c2kv_compress_chunk, ctx, kd, vd, 8, 0, 0) == c2kv.ERR_ARG
    assert _status(c2kv.c2kv_compress_chunk, ctx, kd, vd, 8, 4, 9) == c2kv.ERR_ARG
    assert _status(c2kv.c2kv_compress_chunk, ctx, None, vd, 8, 4, 0) == c2kv.ERR_ARG
    # MEANPOOL needs device memory
    assert _status(c2kv.c2kv_compress_chunk, ctx, kt, vt, 8, 4, 0) == c2kv.ERR_ARG


def test_attend_arg_checks(ctx):
    c2kv = H.lib()
    a = _chunk(ctx)
    cache = c2kv.c2kv_compose(ctx, [0, 1], [a], None, 4)
    q = torch.zeros((2, 1, 4, WL.n_q_heads, WL.head_dim), device="cuda", dtype=torch.bfloat16)
    kv = torch.zeros((2, 1, 4, WL.n_kv_heads, WL.head_dim), device="cuda", dtype=torch.bfloat16)
    out = torch.empty_like(q)
    assert _status(c2kv.c2kv_attend, ctx, cache, -1, q, kv, kv, 5, out) == c2kv.ERR_ARG
    assert _status(c2kv.c2kv_attend, ctx, cache, -1, q, kv, kv, 0, out) == c2kv.ERR_ARG
    assert _status(c2kv.c2kv_attend, ctx, cache, 2, q, kv, kv, 4, out) == c2kv.ERR_ARG
    assert _status(c2kv.c2kv_attend, ctx, cache, -1, None, kv, kv, 4, out) == c2kv.ERR_ARG
    other = H.make_ctx(WL, pool_slots=8)
    try:
        assert _status(c2kv.c2kv_attend, other, cache, -1, q, kv, kv, 4, out) == c2kv.ERR_STATE
        assert _status(c2kv.c2kv_cache_release, other, cache) == c2kv.ERR_STATE
    finally:
        c2kv.c2kv_destroy(other)
    c2kv.c2kv_attend(ctx, cache, -1, q, kv, kv, 4, out)
    c2kv.c2kv_sync(ctx)
    assert torch.isfinite(out.float()).all()
    c2kv.c2kv_cache_release(ctx, cache)
    assert _status(c2kv.c2kv_cache_release, ctx, cache) == c2kv.ERR_STATE


def test_misaligned_pointers_refused(ctx):
    # rows move in 16-byte vectors and by TMA: a misaligned tensor is refused on the host
    c2kv = H.lib()
    a = _chunk(ctx)
    cache = c2kv.c2kv_compose(ctx, [0, 1], [a], None, 4)
    q = torch.zeros((2, 1, 4, WL.n_q_heads, WL.head_dim), device="cuda", dtype=torch.bfloat16)
    kv = torch.zeros((2, 1, 4, WL.n_kv_heads, WL.head_dim), device="cuda", dtype=torch.bfloat16)
    out = torch.empty_like(q)
    lse = torch.empty((2, 1, WL.n_q_heads, 4), device="cuda")
    odd = q.data_ptr() + 2
    assert _status(c2kv.c2kv_attend, ctx, cache, -1, odd, kv, kv, 4, out) == c2kv.ERR_ARG
    assert _status(c2kv.c2kv_attend, ctx, cache, -1, q, kv, kv, 4, out.data_ptr() + 8) == c2kv.ERR_ARG
    assert _status(c2kv.c2kv_attend, ctx, cache, -1, q, kv, kv, 4, out, lse.data_ptr() + 2) == c2kv.ERR_ARG
    assert _status(c2kv.c2kv_attend_noalloc, ctx, cache, -1, odd, kv, kv, 4, out) == c2kv.ERR_ARG
    steps = np.zeros(1, np.int32)
    assert _status(c2kv.c2kv_decode, ctx, cache, -1, odd, kv, kv, steps, out) == c2kv.ERR_ARG
    assert _status(c2kv.c2kv_extract_attention, ctx, 1, odd, kv, kv, 3, 1, out) == c2kv.ERR_ARG
    kt, vt = synth.chunk_tokens(WL, 0, n_tokens=8)
    kd, vd = H.to_dev(kt, WL), H.to_dev(vt, WL)
    assert _status(c2kv.c2kv_compress_chunk, ctx, kd.data_ptr() + 2, vd, 8, 4, 0) == c2kv.ERR_ARG
    # nothing was changed: the aligned call still runs
    c2kv.c2kv_attend(ctx, cache, -1, q, kv, kv, 4, out, lse)
    c2kv.c2kv_sync(ctx)
    assert torch.isfinite(out.float()).all()
    c2kv.c2kv_cache_release(ctx, cache)


def test_device_bounds_check_reports_and_recovers(ctx):
    c2kv = H.lib()
    a = _chunk(ctx)
    c2kv.c2kv_inject_fault(ctx, 1)
    cache = c2kv.c2kv_compose(ctx, [0, 1], [a], None, 4)
    assert _status(c2kv.c2kv_sync, ctx) == c2kv.ERR_DEVICE_BOUNDS
    c2kv.c2kv_cache_release(ctx, cache)
    # the word was cleared and the context still works
    cache = c2kv.c2kv_compose(ctx, [0, 1], [a], None, 4)
    c2kv.c2kv_sync(ctx)
    info = c2kv.c2kv_cache_info(cache)
    pos = c2kv.device_view(info["pos"], (info["rows"],), torch.int32).cpu().numpy()
    assert list(pos[:16]) == [4 * j + 3 for j in range(16)]
    c2kv.c2kv_cache_release(ctx, cache)


def test_destroy_releases_live_caches():
    c2kv = H.lib()
    c = H.make_ctx(WL, pool_slots=64)
    a = _chunk(c)
    for _ in range(3):
        c2kv.c2kv_compose(c, [0, 1], [a], None, 4)
    c2kv.c2kv_destroy(c)          # must free the three caches without error
    assert np.isfinite(1.0)


def test_device_only_calls_refuse_host_memory(ctx):
    # decode and extraction take device tensors only; attend_noalloc takes device or pinned
    # host tensors; pageable host memory (which no kernel may dereference) is refused by all
    # three with ERR_ARG before anything is enqueued
    c2kv = H.lib()
    a = _chunk(ctx)
    cache = c2kv.c2kv_compose(ctx, [0, 1], [a], None, 8)
    q = torch.zeros((2, 1, 4, WL.n_q_heads, WL.head_dim), device="cuda", dtype=torch.bfloat16)
    kv = torch.zeros((2, 1, 4, WL.n_kv_heads, WL.head_dim), device="cuda", dtype=torch.bfloat16)
    out = torch.empty_like(q)
    pageable = torch.zeros(q.shape, dtype=torch.bfloat16)              # torch CPU tensor
    numpy_buf = np.zeros((2, 1, 4, WL.n_kv_heads, WL.head_dim), np.float32)  # 16-byte aligned
    assert numpy_buf.ctypes.data % 16 == 0
    steps = np.zeros(1, np.int32)
    qd = q[:, :, 0].contiguous()
    kd = kv[:, :, 0].contiguous()
    od = torch.empty_like(qd)
    for bad in (torch.zeros(qd.shape, dtype=torch.bfloat16),
                torch.zeros(qd.shape, dtype=torch.bfloat16).pin_memory()):
        assert _status(c2kv.c2kv_decode, ctx, cache, -1, bad, kd, kd, steps, od) == c2kv.ERR_ARG
        assert _status(c2kv.c2kv_decode, ctx, cache, -1, qd, kd, kd, steps, bad) == c2kv.ERR_ARG
    assert _status(c2kv.c2kv_decode, ctx, cache, -1, qd, numpy_buf[:, :, 0].copy(), kd, steps,
                   od) == c2kv.ERR_ARG
    n, k = 3, 1
    xq = torch.zeros((1, 6, WL.n_q_heads, WL.head_dim), device="cuda", dtype=torch.bfloat16)
    xk = torch.zeros((1, 6, WL.n_kv_heads, WL.head_dim), device="cuda", dtype=torch.bfloat16)
    xo = torch.empty_like(xq)
    for bad in (torch.zeros(xq.shape, dtype=torch.bfloat16),
                torch.zeros(xq.shape, dtype=torch.bfloat16).pin_memory()):
        assert _status(c2kv.c2kv_extract_attention, ctx, 1, bad, xk, xk, n, k, xo) == c2kv.ERR_ARG
        assert _status(c2kv.c2kv_extract_attention, ctx, 1, xq, xk, xk, n, k, bad) == c2kv.ERR_ARG
    assert _status(c2kv.c2kv_attend_noalloc, ctx, cache, -1, q, kv, kv, 4, pageable) == c2kv.ERR_ARG
    assert _status(c2kv.c2kv_attend_noalloc, ctx, cache, -1, q, numpy_buf, kv, 4, out) == c2kv.ERR_ARG
    assert "cannot address" in c2kv.c2kv_last_error(ctx)
    # nothing was enqueued, and the context still works
    c2kv.c2kv_decode(ctx, cache, -1, qd, kd, kd, steps, od)
    c2kv.c2kv_extract_attention(ctx, 1, xq, xk, xk, n, k, xo)
    c2kv.c2kv_sync(ctx)
    assert torch.isfinite(od.float()).all() and torch.isfinite(xo.float()).all()
    c2kv.c2kv_cache_release(ctx, cache)
