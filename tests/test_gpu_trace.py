"""Tracing: per-kernel device time through c2kv_profile_enable / c2kv_profile_read."""
import numpy as np
import pytest
import torch

import synth
from tests import _gpu_helpers as H

pytestmark = pytest.mark.gpu


def test_profile_counts_and_times():
    wl = synth.scaled(synth.workload("llama8b"), layers=2, chunks_per_request=3, pool_chunks=3)
    c2kv = H.lib()
    ctx = H.make_ctx(wl, pool_slots=1024)
    try:
        c2kv.c2kv_profile_enable(ctx, True)
        kt, vt = synth.chunk_tokens(wl, 0)
        ids = [c2kv.c2kv_compress_chunk(ctx, H.to_dev(kt, wl), H.to_dev(vt, wl),
                                        wl.chunk_tokens, wl.ratio_k, c2kv.MODE_MEANPOOL)
               for _ in range(3)]
        cache = c2kv.c2kv_compose(ctx, [0, 3], ids, None, wl.n_suffix)
        q, k, v = (H.to_dev(x, wl) for x in synth.suffix(wl))
        out = torch.empty_like(q)
        for _ in range(2):
            c2kv.c2kv_attend(ctx, cache, -1, q, k, v, wl.n_suffix, out)
        prof = c2kv.c2kv_profile_read(ctx)
        assert prof["compress"][1] == 3 and prof["compose"][1] == 1
        assert prof["suffix"][1] == 2 and prof["attention"][1] == 2
        assert all(ms > 0 for ms, n in prof.values() if n)
        assert c2kv.c2kv_profile_read(ctx)["attention"] == (0.0, 0)   # read clears
        c2kv.c2kv_profile_enable(ctx, False)
        c2kv.c2kv_attend(ctx, cache, -1, q, k, v, wl.n_suffix, out)
        assert c2kv.c2kv_profile_read(ctx)["attention"][1] == 0
        assert np.isfinite(out.float().cpu().numpy()).all()
    finally:
        c2kv.c2kv_destroy(ctx)


@pytest.mark.parametrize("split", [False, True], ids=["one_split", "key_range_splits"])
def test_attend_traced_equals_untraced(split):
    # untraced, the attention starts as the suffix kernel's programmatic dependent; traced,
    # events sit between them and they run one after the other: the same O and lse, bit for
    # bit.  With key-range splits the kernel merges them itself (no merge launch), and the
    # merge's counters are back at zero for the next call (three calls in a row agree)
    base = synth.workload("llama8b")
    if split:      # one layer of 3 x 1024 slots, keys split 3 ways
        wl = synth.scaled(base, layers=1, chunks_per_request=3, pool_chunks=3, chunk_tokens=1024,
                          ratio_k=1)
    else:
        wl = synth.scaled(base, layers=2, chunks_per_request=3, pool_chunks=3)
    c2kv = H.lib()
    m = -(-wl.chunk_tokens // wl.ratio_k)
    ctx = H.make_ctx(wl, pool_slots=3 * m + 16, attn_split=3 if split else 0)
    try:
        ids = []
        for cid in range(3):
            kt, vt = synth.chunk_tokens(wl, cid)
            ids.append(c2kv.c2kv_compress_chunk(ctx, H.to_dev(kt, wl), H.to_dev(vt, wl),
                                                wl.chunk_tokens, wl.ratio_k, c2kv.MODE_MEANPOOL))
        cache = c2kv.c2kv_compose(ctx, [0, 3], ids, None, wl.n_suffix)
        q, k, v = (H.to_dev(x, wl) for x in synth.suffix(wl))
        res = []
        for traced in (False, True, False):
            c2kv.c2kv_profile_enable(ctx, traced)
            out = torch.full_like(q, float("nan"))
            lse = torch.full((wl.layers, 1, wl.n_q_heads, wl.n_suffix), float("nan"), device="cuda")
            c2kv.c2kv_attend(ctx, cache, -1, q, k, v, wl.n_suffix, out, lse)
            c2kv.c2kv_sync(ctx)
            res.append((out, lse))
        c2kv.c2kv_profile_enable(ctx, False)
        prof = c2kv.c2kv_profile_read(ctx)
        assert prof["combine"][1] == 0 and prof["attention"][1] == 1
        for o, l in res[1:]:
            assert torch.equal(res[0][0], o) and torch.equal(res[0][1], l)
        assert not torch.isnan(res[0][0]).any()
        c2kv.c2kv_cache_release(ctx, cache)
    finally:
        c2kv.c2kv_destroy(ctx)
