"""c2kv_attend_noalloc: attention for callers that cannot let the library allocate device
memory while they run (an engine that has reserved all of HBM for its own cache pool, a
runtime whose allocator owns every device byte).  It must give the same output as
c2kv_attend -- the call that takes its scratch from the context's memory pool -- and as the
oracle, on two calls in a row (the fixed scratch array keeps the previous call's contents);
refuse requests larger than its fixed 16 MiB array; and take no device memory at its first
call, even under lazy module loading.  This file is named to be collected last."""
import os
import subprocess
import sys
import textwrap

import numpy as np
import pytest
import torch

import synth
from oracle import c2kv_oracle as orc
from tests import _gpu_helpers as H

pytestmark = pytest.mark.gpu

L8B = synth.workload("llama8b")


def _setup(wl, attn_impl=0):
    c2kv = H.lib()
    reqs = synth.requests(wl)
    ids_all = sorted({c for ids, _ in reqs for c in ids})
    chunks = H.oracle_chunks_meanpool(wl, ids_all)
    ctx = H.make_ctx(wl, pool_slots=sum(chunks[c][0].shape[1] for c in ids_all) + 16,
                     attn_impl=attn_impl)
    dev = H.load_stored(ctx, wl, chunks)
    req_ptr = np.cumsum([0] + [len(ids) for ids, _ in reqs])
    cache = c2kv.c2kv_compose(ctx, req_ptr, [dev[c] for ids, _ in reqs for c in ids],
                              [o for _, offs in reqs for o in offs], wl.n_suffix)
    return c2kv, ctx, cache, chunks, reqs


def _check_oracle(got, chunks, reqs, q, k, v, wl, rows):
    for r in rows:
        ids, offs = reqs[r]
        ref = orc.run_request(chunks, ids, offs, q[:, r], k[:, r], v[:, r], wl.rope_theta, wl.dtype)
        H.check_attention(got[:, r], ref["out"], wl, f"noalloc vs oracle, request {r}")


@pytest.mark.parametrize("attn_impl", [0, 1], ids=["tensor_core", "simt"])
def test_noalloc_matches_attend_and_oracle_on_two_calls(attn_impl):
    wl = synth.scaled(L8B, layers=2, chunks_per_request=3, pool_chunks=6, batch=2, draw="distinct",
                      n_suffix=40)
    c2kv, ctx, cache, chunks, reqs = _setup(wl, attn_impl)
    try:
        tol = H.ATTN_TOL[wl.dtype]
        for seed in (11, 12):                     # two calls in a row, different inputs
            qn, kn, vn = synth.suffix(wl, seed)
            q, k, v = (H.to_dev(x, wl) for x in (qn, kn, vn))
            ref = torch.empty_like(q)
            ref_lse = torch.empty((wl.layers, wl.batch, wl.n_q_heads, wl.n_suffix), device="cuda")
            c2kv.c2kv_attend(ctx, cache, -1, q, k, v, wl.n_suffix, ref, ref_lse)
            got = torch.full_like(q, float("nan"))
            got_lse = torch.full_like(ref_lse, float("nan"))
            c2kv.c2kv_attend_noalloc(ctx, cache, -1, q, k, v, wl.n_suffix, got, got_lse)
            c2kv.c2kv_sync(ctx)
            r = ref.double().cpu().numpy()
            g = got.double().cpu().numpy()
            assert np.isfinite(g).all()
            assert np.all(np.abs(g - r) <= tol + tol * np.abs(r))
            assert torch.allclose(got_lse, ref_lse, atol=1e-4, rtol=1e-5)
            _check_oracle(g, chunks, reqs, qn, kn, vn, wl, range(wl.batch))
    finally:
        c2kv.c2kv_destroy(ctx)


def test_noalloc_f32_matches_attend_and_oracle():
    wl = synth.workload("tiny_f32")
    c2kv, ctx, cache, chunks, reqs = _setup(wl)
    try:
        qn, kn, vn = synth.suffix(wl, 4)
        q, k, v = (H.to_dev(x, wl) for x in (qn, kn, vn))
        ref, got = torch.empty_like(q), torch.empty_like(q)
        for _ in range(2):
            c2kv.c2kv_attend(ctx, cache, -1, q, k, v, wl.n_suffix, ref)
            c2kv.c2kv_attend_noalloc(ctx, cache, -1, q, k, v, wl.n_suffix, got)
        c2kv.c2kv_sync(ctx)
        H.check_attention(got.double().cpu().numpy(), ref.double().cpu().numpy(), wl, "f32 vs attend")
        _check_oracle(got.double().cpu().numpy(), chunks, reqs, qn, kn, vn, wl, [0])
    finally:
        c2kv.c2kv_destroy(ctx)


def test_noalloc_more_requests_than_one_launch_takes():
    # 257 requests: the suffix and attention kernels take at most 256 requests a launch, so
    # the call launches twice over the one scratch array
    wl = synth.scaled(L8B, layers=1, n_q_heads=8, n_kv_heads=2, chunk_tokens=16, ratio_k=4,
                      chunks_per_request=1, pool_chunks=257, batch=257, draw="distinct", n_suffix=3)
    c2kv, ctx, cache, chunks, reqs = _setup(wl)
    try:
        qn, kn, vn = synth.suffix(wl, 6)
        q, k, v = (H.to_dev(x, wl) for x in (qn, kn, vn))
        ref, got = torch.empty_like(q), torch.full_like(q, float("nan"))
        c2kv.c2kv_attend(ctx, cache, -1, q, k, v, wl.n_suffix, ref)
        c2kv.c2kv_attend_noalloc(ctx, cache, -1, q, k, v, wl.n_suffix, got)
        c2kv.c2kv_sync(ctx)
        g = got.double().cpu().numpy()
        H.check_attention(g, ref.double().cpu().numpy(), wl, "257 requests vs attend")
        _check_oracle(g, chunks, reqs, qn, kn, vn, wl, [0, 255, 256])
    finally:
        c2kv.c2kv_destroy(ctx)


def test_noalloc_pinned_host_tensors_in_place():
    # suffix inputs and outputs in pinned host memory: read and written in place over the link
    wl = synth.scaled(L8B, layers=2, chunks_per_request=2, pool_chunks=2, n_suffix=24)
    c2kv, ctx, cache, chunks, reqs = _setup(wl)
    try:
        qn, kn, vn = synth.suffix(wl, 8)
        qd, kd, vd = (H.to_dev(x, wl) for x in (qn, kn, vn))
        qh, kh, vh = (x.cpu().pin_memory() for x in (qd, kd, vd))
        ref = torch.empty_like(qd)
        out_h = torch.full(qd.shape, float("nan"), dtype=qd.dtype).pin_memory()
        lse_h = torch.full((wl.layers, 1, wl.n_q_heads, wl.n_suffix), float("nan")).pin_memory()
        ref_lse = torch.empty(lse_h.shape, device="cuda")
        c2kv.c2kv_attend(ctx, cache, -1, qd, kd, vd, wl.n_suffix, ref, ref_lse)
        c2kv.c2kv_attend_noalloc(ctx, cache, -1, qh, kh, vh, wl.n_suffix, out_h, lse_h)
        c2kv.c2kv_sync(ctx)
        g = out_h.double().numpy()
        H.check_attention(g, ref.double().cpu().numpy(), wl, "host tensors vs attend")
        assert torch.allclose(lse_h, ref_lse.cpu(), atol=1e-4, rtol=1e-5)
        _check_oracle(g, chunks, reqs, qn, kn, vn, wl, [0])
    finally:
        c2kv.c2kv_destroy(ctx)


def test_noalloc_single_layer_and_size_limit():
    wl = synth.scaled(L8B, layers=32, chunks_per_request=2, pool_chunks=2, n_suffix=80)
    c2kv, ctx, cache, chunks, reqs = _setup(wl)
    try:
        q, k, v = (H.to_dev(x, wl) for x in synth.suffix(wl, 3))
        # one layer at a time fits the fixed array
        ref = torch.empty_like(q[5])
        got = torch.empty_like(q[5])
        c2kv.c2kv_attend(ctx, cache, 5, q[5], k[5], v[5], wl.n_suffix, ref)
        c2kv.c2kv_attend_noalloc(ctx, cache, 5, q[5], k[5], v[5], wl.n_suffix, got)
        c2kv.c2kv_sync(ctx)
        tol = H.ATTN_TOL[wl.dtype]
        r, g = ref.double().cpu().numpy(), got.double().cpu().numpy()
        assert np.all(np.abs(g - r) <= tol + tol * np.abs(r))
        # all 32 layers x 80 tokens x 32 heads x 128 x 2 B = 20 MiB > 16 MiB: refused
        out = torch.empty_like(q)
        with pytest.raises(c2kv.C2KVError) as ei:
            c2kv.c2kv_attend_noalloc(ctx, cache, -1, q, k, v, wl.n_suffix, out)
        assert ei.value.status == c2kv.ERR_ARG and "16 MiB" in str(ei.value)
        c2kv.c2kv_sync(ctx)           # nothing was enqueued by the refused call
    finally:
        c2kv.c2kv_destroy(ctx)


_FIRST_CALL = textwrap.dedent("""
    import sys
    sys.path.insert(0, {root!r})
    import numpy as np, torch
    import synth
    from tests import _gpu_helpers as H
    c2kv = H.lib()
    wl = synth.scaled(synth.workload("llama8b"), layers=2, chunks_per_request=2, pool_chunks=2,
                      n_suffix=16)
    reqs = synth.requests(wl)
    chunks = H.oracle_chunks_meanpool(wl, [0, 1])
    ctx = H.make_ctx(wl, pool_slots=512)
    dev = H.load_stored(ctx, wl, chunks)
    (ids, offs), = reqs
    cache = c2kv.c2kv_compose(ctx, [0, 2], [dev[c] for c in ids], offs, wl.n_suffix)
    q, k, v = (H.to_dev(x, wl) for x in synth.suffix(wl, 1))
    out = torch.empty_like(q)
    c2kv.c2kv_sync(ctx)
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    c2kv.c2kv_attend_noalloc(ctx, cache, -1, q, k, v, wl.n_suffix, out)
    c2kv.c2kv_sync(ctx)
    free1 = torch.cuda.mem_get_info()[0]
    assert torch.isfinite(out.float()).all()
    print("FREE_DELTA", free0 - free1)
""")


def test_noalloc_first_call_takes_no_device_memory_under_lazy_loading():
    # A fresh process with lazy module loading: c2kv_create must already have reserved the
    # fixed array and loaded the kernels, so the device's free memory is the same before and
    # after the first c2kv_attend_noalloc call.
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    env = dict(os.environ, CUDA_MODULE_LOADING="LAZY")
    res = subprocess.run([sys.executable, "-c", _FIRST_CALL.format(root=root)], env=env,
                         capture_output=True, text=True, timeout=240, cwd=root)
    assert res.returncode == 0, res.stdout[-2000:] + res.stderr[-2000:]
    delta = [int(line.split()[1]) for line in res.stdout.splitlines() if line.startswith("FREE_DELTA")]
    assert delta == [0], res.stdout[-2000:]
