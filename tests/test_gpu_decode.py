"""Decode attention (one new token per request after the suffix) against the oracle's
decode step: every composed slot and suffix rows 0 .. step as keys, one query row."""
import numpy as np
import pytest
import torch

import synth
from oracle import c2kv_oracle as orc
from tests import _gpu_helpers as H

pytestmark = pytest.mark.gpu

L8B_1 = synth.scaled(synth.workload("llama8b"), layers=1)
TINY = synth.workload("tiny_f32")


def _small(wl, **kw):
    base = dict(batch=1, chunks_per_request=3, pool_chunks=3, chunk_tokens=256)
    base.update(kw)
    return synth.scaled(wl, **base)


def _decode_case(wl, steps, prefill=None, layer=-1, extra_steps=0, attn_impl=0):
    """Compose the workload's requests, optionally run c2kv_attend over `prefill` suffix
    tokens, then decode: request r's new token at suffix index steps[r] (and, with
    extra_steps, the following steps one call at a time).  Every decode output and lse is
    compared with the oracle's decode step for that request.  attn_impl 0 lets the library
    pick the route (the tensor-core kernel for these sizes with bf16), C2KV_ATTN_SIMT forces
    the CUDA-core decode kernel."""
    c2kv = H.lib()
    reqs = synth.requests(wl)
    B = len(reqs)
    n_tok = max(steps) + extra_steps + 1
    wl_s = synth.scaled(wl, n_suffix=n_tok)
    all_ids = sorted({c for ids, _ in reqs for c in ids})
    chunks = H.oracle_chunks_meanpool(wl, all_ids)
    pool = sum(orc.n_slots(wl.chunk_tokens, wl.ratio_k) for _ in all_ids) + 16
    ctx = H.make_ctx(wl, pool_slots=pool, attn_impl=attn_impl)
    try:
        dev = H.load_stored(ctx, wl, chunks)
        req_ptr = np.cumsum([0] + [len(ids) for ids, _ in reqs])
        cache = c2kv.c2kv_compose(ctx, req_ptr, [dev[c] for ids, _ in reqs for c in ids],
                                  [o for _, offs in reqs for o in offs], suffix_capacity=n_tok)
        q, ks, vs = synth.suffix(wl_s, layers=wl.layers)          # [L, B, n_tok, H, d]
        q, ks, vs = q[:, :B], ks[:, :B], vs[:, :B]
        lsel = slice(None) if layer == -1 else slice(layer, layer + 1)
        if prefill:
            # write suffix tokens 0 .. prefill-1 with the suffix attention
            qd, kd, vd = (H.to_dev(x[lsel, :, :prefill], wl) for x in (q, ks, vs))
            out = torch.empty_like(qd)
            c2kv.c2kv_attend(ctx, cache, layer, qd, kd, vd, prefill, out)
        oracle = [orc.compose(chunks, ids, offs, wl.rope_theta, wl.dtype) for ids, offs in reqs]
        st = np.asarray(steps)
        for extra in range(extra_steps + 1):
            cur = st + extra
            pick = lambda x: np.stack([x[:, b, cur[b]] for b in range(B)], axis=1)  # [L, B, H, d]
            qd, kd, vd = (H.to_dev(pick(x)[lsel], wl) for x in (q, ks, vs))
            out = torch.full_like(qd, float("nan"))
            lse = torch.full(qd.shape[:-1], float("nan"), device="cuda")
            c2kv.c2kv_decode(ctx, cache, layer, qd, kd, vd, cur, out, lse)
            c2kv.c2kv_sync(ctx)
            got = out.double().cpu().numpy()
            got_lse = lse.double().cpu().numpy()
            for b in range(B):
                k_c, v_c, _, l_req = oracle[b]
                t = int(cur[b])
                o, l_ = orc.decode_step(k_c[lsel], v_c[lsel], l_req, ks[lsel, b, :t], vs[lsel, b, :t],
                                        q[lsel, b, t], ks[lsel, b, t], vs[lsel, b, t], t,
                                        wl.rope_theta, wl.dtype)
                H.check_attention(got[:, b], o, wl, f"decode O req {b} step {t}")
                assert np.allclose(got_lse[:, b], l_, atol=1e-3, rtol=1e-4), f"lse req {b} step {t}"
        # the decode token's position was recorded with its row
        info, gk, gv, gpos = H.cache_arrays(cache, wl)
        for b in range(B):
            base, s = info["row_base"][b], info["n_slots"][b]
            last = int(st[b]) + extra_steps
            assert gpos[base + s + last] == oracle[b][3] + last
        c2kv.c2kv_cache_release(ctx, cache)
    finally:
        c2kv.c2kv_destroy(ctx)


IMPLS = pytest.mark.parametrize("impl", [0, 1], ids=["auto", "cuda_core"])   # 1: C2KV_ATTN_SIMT
TC = 2                                                                          # C2KV_ATTN_TC


@IMPLS
def test_decode_after_suffix_attention(impl):
    # the suffix of 16 tokens written by attend, then the 17th token decoded
    _decode_case(_small(L8B_1, layers=2), steps=[16], prefill=16, attn_impl=impl)


@IMPLS
def test_decode_sequence_from_step0(impl):
    # straight after compose: steps 0, 1, 2, 3 one call at a time
    _decode_case(_small(L8B_1, layers=2), steps=[0], extra_steps=3, attn_impl=impl)


@IMPLS
def test_decode_batched_ragged_steps(impl):
    wl = _small(synth.workload("batched"), batch=3, chunks_per_request=4, pool_chunks=32)
    _decode_case(wl, steps=[5, 0, 11], prefill=12, attn_impl=impl)


def test_decode_at_tile_edges():
    # new tokens at the last row of a 128-row key tile and at the first two of the next
    # (slots + step + 1 = 256, 257, 258): the rows after the new token up to the next tile's
    # edge hold no data until the step zeroes them
    wl = _small(L8B_1, layers=2, chunk_tokens=256, ratio_k=4, chunks_per_request=3)
    s = 3 * 64
    _decode_case(wl, steps=[256 - s - 1], prefill=256 - s - 1, extra_steps=2)


def test_decode_single_layer_of_many():
    _decode_case(_small(L8B_1, layers=3), steps=[7], prefill=8, layer=1)


def test_decode_f32_tiny():
    _decode_case(TINY, steps=[4], prefill=5)


@IMPLS
def test_decode_long_context_splits(impl):
    # 32 chunks x 1024 tokens at k=4: 8192 slots, so the key range is split over many CTAs
    # and merged
    wl = _small(L8B_1, chunk_tokens=1024, ratio_k=4, chunks_per_request=32, pool_chunks=32)
    _decode_case(wl, steps=[3], prefill=3, attn_impl=impl)


@pytest.mark.parametrize("noalloc", [False, True], ids=["attend", "attend_noalloc"])
def test_decode_keeps_rows_written_by_attend(noalloc):
    # a suffix of 40 tokens written by attention, then a decode step at suffix index 5 (the
    # sequence taken back to that point): rows 6 .. 39 keep what the attention wrote, the
    # zeroing for whole key tiles never reaching rows a call wrote
    c2kv = H.lib()
    wl = _small(L8B_1, layers=2)
    reqs = synth.requests(wl)
    all_ids = sorted({c for ids, _ in reqs for c in ids})
    chunks = H.oracle_chunks_meanpool(wl, all_ids)
    pool = sum(orc.n_slots(wl.chunk_tokens, wl.ratio_k) for _ in all_ids) + 16
    ctx = H.make_ctx(wl, pool_slots=pool)
    try:
        dev = H.load_stored(ctx, wl, chunks)
        req_ptr = np.cumsum([0] + [len(ids) for ids, _ in reqs])
        cache = c2kv.c2kv_compose(ctx, req_ptr, [dev[c] for ids, _ in reqs for c in ids],
                                  [o for _, offs in reqs for o in offs], suffix_capacity=64)
        q, ks, vs = synth.suffix(synth.scaled(wl, n_suffix=40), layers=wl.layers)
        qd, kd, vd = (H.to_dev(x, wl) for x in (q, ks, vs))
        attend = c2kv.c2kv_attend_noalloc if noalloc else c2kv.c2kv_attend
        attend(ctx, cache, -1, qd, kd, vd, 40, torch.empty_like(qd))
        c2kv.c2kv_sync(ctx)
        info, k0, v0, _ = H.cache_arrays(cache, wl)
        base, s = info["row_base"][0], info["n_slots"][0]
        pick = [H.to_dev(x[:, :, 5], wl) for x in (q, ks, vs)]
        out = torch.empty_like(pick[0])
        c2kv.c2kv_decode(ctx, cache, -1, pick[0], pick[1], pick[2], [5], out)
        c2kv.c2kv_sync(ctx)
        _, k1, v1, _ = H.cache_arrays(cache, wl)
        rows = slice(base + s + 6, base + s + 40)
        assert np.array_equal(k1[:, rows], k0[:, rows]) and np.array_equal(v1[:, rows], v0[:, rows])
        assert np.isfinite(out.float().cpu().numpy()).all()
        c2kv.c2kv_cache_release(ctx, cache)
    finally:
        c2kv.c2kv_destroy(ctx)


@pytest.mark.parametrize("long", [False, True])
def test_decode_traced_equals_untraced(long):
    # untraced, the decode kernel is the suffix kernel's programmatic dependent and loads the
    # tiles before the new row while that kernel runs; traced, the two run one after the
    # other.  The same step decoded both ways (the new row rewritten with the same bits):
    # the same output and lse, bit for bit; long: key-range splits and their merge
    c2kv = H.lib()
    if long:
        wl = _small(L8B_1, chunk_tokens=1024, ratio_k=4, chunks_per_request=32, pool_chunks=32)
    else:
        wl = _small(synth.workload("batched"), batch=3, chunks_per_request=4, pool_chunks=32,
                    layers=2)
    reqs = synth.requests(wl)
    B = len(reqs)
    steps = [4 + 3 * b for b in range(B)]
    n_tok = max(steps) + 1
    all_ids = sorted({c for ids, _ in reqs for c in ids})
    chunks = H.oracle_chunks_meanpool(wl, all_ids)
    pool = sum(orc.n_slots(wl.chunk_tokens, wl.ratio_k) for _ in all_ids) + 16
    ctx = H.make_ctx(wl, pool_slots=pool)
    try:
        dev = H.load_stored(ctx, wl, chunks)
        req_ptr = np.cumsum([0] + [len(ids) for ids, _ in reqs])
        cache = c2kv.c2kv_compose(ctx, req_ptr, [dev[c] for ids, _ in reqs for c in ids],
                                  [o for _, offs in reqs for o in offs], suffix_capacity=n_tok)
        q, ks, vs = synth.suffix(synth.scaled(wl, n_suffix=n_tok), layers=wl.layers)
        q, ks, vs = q[:, :B], ks[:, :B], vs[:, :B]
        pre = min(steps)
        qd, kd, vd = (H.to_dev(x[:, :, :pre], wl) for x in (q, ks, vs))
        c2kv.c2kv_attend(ctx, cache, -1, qd, kd, vd, pre, torch.empty_like(qd))
        for b in range(B):        # suffix rows pre .. steps[b]-1 of each request, one at a time
            for t in range(pre, steps[b]):
                cur = [t if r == b else steps[r] for r in range(B)]
                pick = [np.stack([x[:, r, cur[r]] for r in range(B)], axis=1) for x in (q, ks, vs)]
                qd, kd, vd = (H.to_dev(x, wl) for x in pick)
                c2kv.c2kv_decode(ctx, cache, -1, qd, kd, vd, cur, torch.empty_like(qd))
        pick = [np.stack([x[:, r, steps[r]] for r in range(B)], axis=1) for x in (q, ks, vs)]
        qd, kd, vd = (H.to_dev(x, wl) for x in pick)
        res = []
        for traced in (False, True):
            c2kv.c2kv_profile_enable(ctx, traced)
            out = torch.full_like(qd, float("nan"))
            lse = torch.full(qd.shape[:-1], float("nan"), device="cuda")
            c2kv.c2kv_decode(ctx, cache, -1, qd, kd, vd, steps, out, lse)
            c2kv.c2kv_sync(ctx)
            res.append((out, lse))
        c2kv.c2kv_profile_enable(ctx, False)
        assert c2kv.c2kv_profile_read(ctx)["decode"][1] >= 1
        assert torch.equal(res[0][0], res[1][0])
        assert torch.equal(res[0][1], res[1][1])
        assert not torch.isnan(res[0][0]).any()
        c2kv.c2kv_cache_release(ctx, cache)
    finally:
        c2kv.c2kv_destroy(ctx)


def test_decode_gqa8_and_mha():
    _decode_case(_small(synth.workload("long70b"), batch=1, chunks_per_request=4,
                        pool_chunks=4), steps=[2], prefill=2)
    _decode_case(_small(L8B_1, n_q_heads=8, n_kv_heads=8), steps=[1], prefill=1)


def test_decode_rejects_bad_steps_and_layouts():
    c2kv = H.lib()
    wl = _small(L8B_1)
    ctx = H.make_ctx(wl, pool_slots=1024)
    try:
        chunks = H.oracle_chunks_meanpool(wl, [0])
        dev = H.load_stored(ctx, wl, chunks)
        cache = c2kv.c2kv_compose(ctx, [0, 1], [dev[0]], [0], suffix_capacity=4)
        q = torch.zeros((1, 1, wl.n_q_heads, wl.head_dim), dtype=torch.bfloat16, device="cuda")
        kv = torch.zeros((1, 1, wl.n_kv_heads, wl.head_dim), dtype=torch.bfloat16, device="cuda")
        for bad in ([4], [-1]):                      # outside [0, suffix_capacity)
            with pytest.raises(c2kv.C2KVError) as ei:
                c2kv.c2kv_decode(ctx, cache, -1, q, kv, kv, bad, torch.empty_like(q))
            assert ei.value.status == c2kv.ERR_ARG
        with pytest.raises(c2kv.C2KVError) as ei:
            c2kv.c2kv_decode(ctx, cache, 5, q, kv, kv, [0], torch.empty_like(q))
        assert ei.value.status == c2kv.ERR_ARG
    finally:
        c2kv.c2kv_destroy(ctx)
    wl3 = _small(L8B_1, n_q_heads=6, n_kv_heads=2)   # G = 3
    ctx = H.make_ctx(wl3, pool_slots=1024)
    try:
        chunks = H.oracle_chunks_meanpool(wl3, [0])
        dev = H.load_stored(ctx, wl3, chunks)
        cache = c2kv.c2kv_compose(ctx, [0, 1], [dev[0]], [0], suffix_capacity=4)
        q = torch.zeros((1, 1, 6, wl3.head_dim), dtype=torch.bfloat16, device="cuda")
        kv = torch.zeros((1, 1, 2, wl3.head_dim), dtype=torch.bfloat16, device="cuda")
        with pytest.raises(c2kv.C2KVError) as ei:
            c2kv.c2kv_decode(ctx, cache, -1, q, kv, kv, [0], torch.empty_like(q))
        assert ei.value.status == c2kv.ERR_UNSUPPORTED
    finally:
        c2kv.c2kv_destroy(ctx)


@pytest.mark.parametrize("impl", [TC, 1], ids=["tensor_cores", "cuda_core"])
def test_decode_more_requests_than_one_launch_takes(impl):
    # 260 requests: the attention kernels take at most 256 requests a launch, so the step runs
    # as two groups (on the tensor-core route its split partials are merged once, after the
    # last group); every request's output against the oracle
    wl = _small(synth.workload("batched"), batch=260, chunks_per_request=1, pool_chunks=260,
                chunk_tokens=64, layers=1, draw="distinct")
    _decode_case(wl, steps=[2 + (b % 5) for b in range(260)], prefill=7, attn_impl=impl)
