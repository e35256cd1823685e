"""c2kv_attend_noalloc: attention for callers that cannot let the library allocate device
memory while they run (an engine that has reserved all of HBM for its own cache pool, a
runtime whose allocator owns every device byte).  It must give the same output as
c2kv_attend -- the call that takes its scratch from the context's memory pool -- on two
calls in a row (the fixed scratch array keeps the previous call's contents), and refuse
requests larger than its fixed 16 MiB array.  This file is named to be collected last."""
import numpy as np
import pytest
import torch

import synth
from tests import _gpu_helpers as H

pytestmark = pytest.mark.gpu


def _setup(wl):
    c2kv = H.lib()
    reqs = synth.requests(wl)
    ids_all = sorted({c for ids, _ in reqs for c in ids})
    chunks = H.oracle_chunks_meanpool(wl, ids_all)
    ctx = H.make_ctx(wl, pool_slots=4096)
    dev = H.load_stored(ctx, wl, chunks)
    req_ptr = np.cumsum([0] + [len(ids) for ids, _ in reqs])
    cache = c2kv.c2kv_compose(ctx, req_ptr, [dev[c] for ids, _ in reqs for c in ids],
                              [o for _, offs in reqs for o in offs], wl.n_suffix)
    return c2kv, ctx, cache


@pytest.mark.parametrize("attn_impl", [0, 1], ids=["tensor_core", "simt"])
def test_noalloc_matches_attend_on_two_calls(attn_impl):
    wl = synth.scaled(synth.workload("llama8b"), layers=2, chunks_per_request=3,
                      pool_chunks=3, batch=2, draw="distinct", n_suffix=40)
    c2kv, ctx, cache = _setup(synth.scaled(wl, batch=2))
    try:
        tol = H.ATTN_TOL[wl.dtype]
        for seed in (11, 12):                     # two calls in a row, different inputs
            q, k, v = (H.to_dev(x, wl) for x in synth.suffix(wl, seed))
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
    finally:
        c2kv.c2kv_destroy(ctx)


def test_noalloc_single_layer_and_size_limit():
    wl = synth.scaled(synth.workload("llama8b"), layers=32, chunks_per_request=2,
                      pool_chunks=2, n_suffix=80)
    c2kv, ctx, cache = _setup(wl)
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
