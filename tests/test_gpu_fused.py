"""Fused compose + attend (c2kv_compose_attend) against the oracle, and against the unfused
calls it replaces: the output, the normaliser and the whole composed cache it leaves behind
(turned K within one storage ulp, V and positions bit-exact, suffix rows as attend writes
them)."""
import numpy as np
import pytest
import torch

import synth
from oracle import c2kv_oracle as orc
from tests import _gpu_helpers as H

pytestmark = pytest.mark.gpu

L8B = synth.workload("llama8b")


def _run(ctx, wl, dev, reqs, q, ks, vs, sq, fused, host_io=False):
    """compose_attend (fused=True) or compose + attend; returns (cache, out, lse) on the
    device.  host_io: the suffix tensors, O and lse live in pinned host memory."""
    c2kv = H.lib()
    B = len(reqs)
    req_ptr = np.cumsum([0] + [len(ids) for ids, _ in reqs])
    flat = [dev[c] for ids, _ in reqs for c in ids]
    offs = [o for _, o_ in reqs for o in o_]
    qd, kd, vd = (H.to_dev(x, wl) for x in (q, ks, vs))
    if host_io:
        qd, kd, vd = (x.cpu().pin_memory() for x in (qd, kd, vd))
        out = torch.empty(qd.shape, dtype=qd.dtype, pin_memory=True).fill_(float("nan"))
        lse = torch.empty((wl.layers, B, wl.n_q_heads, sq), pin_memory=True).fill_(float("nan"))
    else:
        out = torch.full_like(qd, float("nan"))
        lse = torch.full((wl.layers, B, wl.n_q_heads, sq), float("nan"), device="cuda")
    if fused:
        cache = c2kv.c2kv_compose_attend(ctx, req_ptr, flat, offs, sq, qd, kd, vd, sq, out, lse)
    else:
        cache = c2kv.c2kv_compose(ctx, req_ptr, flat, offs, suffix_capacity=sq)
        c2kv.c2kv_attend(ctx, cache, -1, qd, kd, vd, sq, out, lse)
    c2kv.c2kv_sync(ctx)
    if host_io:
        out, lse = out.cuda(), lse.cuda()
    return cache, out, lse


def _fused_case(wl, reqs=None, n_suffix=None, attn_split=0, host=(), fixed_pos=False,
                compare_unfused=True, fuse=2, host_io=False, attn_pairs=0):
    """compose_attend with the fused kernel forced (fuse=2) unless it cannot take the call,
    checked against the oracle and, bit for bit, against compose + attend."""
    c2kv = H.lib()
    sq = wl.n_suffix if n_suffix is None else n_suffix
    wl = synth.scaled(wl, n_suffix=sq)
    reqs = synth.requests(wl) if reqs is None else reqs
    all_ids = sorted({c for ids, _ in reqs for c in ids})
    chunks = H.oracle_chunks_meanpool(wl, all_ids)
    pool = sum(chunks[c][0].shape[1] for c in all_ids) + 16
    ctx = H.make_ctx(wl, pool_slots=pool, attn_split=attn_split, fixed_pos=int(fixed_pos),
                     fuse=fuse, attn_pairs=attn_pairs)
    keep = []
    try:
        dev = H.load_stored(ctx, wl, chunks, host=host, keep=keep)
        B = len(reqs)
        q, ks, vs = synth.suffix(synth.scaled(wl, batch=max(B, wl.batch)), layers=wl.layers)
        q, ks, vs = q[:, :B], ks[:, :B], vs[:, :B]
        cache, out, lse = _run(ctx, wl, dev, reqs, q, ks, vs, sq, fused=True, host_io=host_io)
        info, gk, gv, gpos = H.cache_arrays(cache, wl)
        got = out.double().cpu().numpy()
        got_lse = lse.double().cpu().numpy()
        for r, (ids, offs) in enumerate(reqs):
            if ids:
                ref = orc.run_request(chunks, ids, offs, q[:, r], ks[:, r], vs[:, r],
                                      wl.rope_theta, wl.dtype, fixed_pos=fixed_pos)
            else:                              # no composed slot: attention over the suffix
                none = np.zeros((wl.layers, 0, wl.n_kv_heads, wl.head_dim))
                o, ls = orc.attend(none, none, 0, q[:, r], ks[:, r], vs[:, r], wl.rope_theta,
                                   wl.dtype)
                ref = dict(out=o, lse=ls, l_req=0)
            H.check_attention(got[:, r], ref["out"], wl, f"O req {r}")
            assert np.allclose(got_lse[:, r], ref["lse"], atol=1e-3, rtol=1e-4), "lse"
            base, s = info["row_base"][r], info["n_slots"][r]
            if ids:
                ok, ov, opos, _ = orc.compose(chunks, ids, offs, wl.rope_theta, wl.dtype, fixed_pos)
                assert np.array_equal(gpos[base:base + s], opos)               # bit-exact
                assert np.array_equal(gv[:, base:base + s], ov)                # bit-exact
                stored = np.concatenate([chunks[c][0] for c in ids], axis=1)
                H.check_rotated(gk[:, base:base + s], ok, stored, wl, f"fused cache K req {r}")
            assert np.array_equal(gpos[base + s: base + s + sq],
                                  orc.suffix_positions(ref["l_req"], sq))
            assert np.array_equal(gv[:, base + s: base + s + sq], vs[:, r].astype(np.float64))
        if compare_unfused:
            cache_u, out_u, lse_u = _run(ctx, wl, dev, reqs, q, ks, vs, sq, fused=False)
            info_u, uk, uv, upos = H.cache_arrays(cache_u, wl)
            # the same stored slots turned by the same arithmetic: the same bits, over every
            # row either call writes (slots, suffix, and the zeroed rows up to the tile edge)
            for r in range(B):
                base, s = info["row_base"][r], info["n_slots"][r]
                assert info_u["row_base"][r] == base and info_u["n_slots"][r] == s
                assert np.array_equal(gpos[base:base + s + sq], upos[base:base + s + sq])
                end = base + (s + sq + 127) // 128 * 128
                assert np.array_equal(gk[:, base:end], uk[:, base:end])
                assert np.array_equal(gv[:, base:end], uv[:, base:end])
            assert torch.equal(out, out_u)
            assert torch.equal(lse, lse_u)
            c2kv.c2kv_cache_release(ctx, cache_u)
        c2kv.c2kv_cache_release(ctx, cache)
    finally:
        c2kv.c2kv_destroy(ctx)


def test_fused_llama8b_two_layers():
    # 10 chunks of 128 slots: every key tile comes from one occurrence
    _fused_case(synth.scaled(L8B, layers=2))


def test_fused_gqa8_tiles_across_occurrences():
    # 64 slots per chunk: every key tile holds two occurrences, each turned by its own offset
    _fused_case(synth.scaled(synth.workload("long70b"), chunks_per_request=5, pool_chunks=8,
                             n_suffix=48))


def test_fused_batched_duplicates():
    _fused_case(synth.scaled(synth.workload("batched"), batch=3, chunks_per_request=4,
                             pool_chunks=32, n_suffix=40))


def test_fused_ragged_gaps_and_empty_request():
    wl = synth.scaled(L8B, layers=2, chunk_tokens=300, ratio_k=10, pool_chunks=4, n_suffix=37)
    reqs = [([0, 2, 1], [5, 400, 900]),        # gaps between occurrences
            ([], []),                          # reuses no chunk: every key from the cache
            ([3, 3], [0, 300]),                # the same chunk twice
            ([1], [0])]
    _fused_case(wl, reqs=reqs)


def test_fused_uncompressed_long_chunk():
    # k = 1: 700 slots of one occurrence over six key tiles
    wl = synth.scaled(L8B, layers=1, chunk_tokens=700, ratio_k=1, chunks_per_request=1,
                      pool_chunks=1, n_suffix=20)
    _fused_case(wl)


def test_fused_long_suffix_across_tiles():
    # 225 composed slots, 300 suffix tokens: the suffix starts inside tile 1, fills tiles 2
    # and 3 (whole tiles from the suffix tensors) and ends inside tile 4, whose rows past it
    # are zeros; five pairs of query tiles, the last of which writes the cache
    wl = synth.scaled(L8B, layers=2, chunk_tokens=300, ratio_k=4, chunks_per_request=3,
                      pool_chunks=3, n_suffix=300)
    _fused_case(wl)


@pytest.mark.parametrize("group", [1, 2, 16])
def test_fused_query_head_groups(group):
    # G query heads per KV head: a Q tile packs 128 / G tokens, so the suffix preparation's
    # items (token, chunk pair) turn G rows each; 2 KV heads keep the case small
    wl = synth.scaled(L8B, layers=2, n_q_heads=2 * group, n_kv_heads=2, chunk_tokens=300,
                      ratio_k=4, chunks_per_request=3, pool_chunks=3, n_suffix=50)
    _fused_case(wl)


@pytest.mark.parametrize("n_suffix", [1, 128, 129])
def test_fused_suffix_at_tile_edges(n_suffix):
    # 256 composed slots (two whole tiles): a suffix of 128 is one whole suffix tile (V by a
    # 128-row box, K' by cp.async), 129 adds a tile of one suffix row and 127 zero rows, 1 is
    # a tile of one row
    wl = synth.scaled(L8B, layers=2, chunk_tokens=512, ratio_k=4, chunks_per_request=2,
                      pool_chunks=2, n_suffix=n_suffix)
    _fused_case(wl)


@pytest.mark.parametrize("per_cta", [2, 3])
def test_attend_pairs_run_in_turn(per_cta):
    # compose, then attention with several pairs of query tiles per CTA: 200 suffix tokens
    # are 7 query tiles, i.e. 4 pairs, the last without a tile B
    wl = synth.scaled(L8B, layers=2, chunk_tokens=300, ratio_k=4, chunks_per_request=3,
                      pool_chunks=3, n_suffix=200)
    _fused_case(wl, fuse=1, attn_pairs=per_cta)


@pytest.mark.parametrize("split", [2, 5])
def test_fused_key_range_splits(split):
    wl = synth.scaled(L8B, layers=1, chunk_tokens=512, ratio_k=2, chunks_per_request=3,
                      pool_chunks=3, n_suffix=70)
    _fused_case(wl, attn_split=split)


def test_fused_fixed_pos():
    wl = synth.scaled(L8B, layers=1, chunks_per_request=3, pool_chunks=3, n_suffix=16)
    _fused_case(wl, fixed_pos=True)


def test_compose_attend_unfused_routes():
    # fp32 (CUDA-core attention) and host-resident chunks take compose, then attend
    _fused_case(synth.workload("tiny_f32"))
    wl = synth.scaled(L8B, layers=1, chunks_per_request=3, pool_chunks=3, n_suffix=16)
    _fused_case(wl, host={0, 2})


@pytest.mark.parametrize("layers", [2, 5])
def test_compose_attend_host_chunks_pipelined(layers):
    # host-resident chunks over several layers: composed in layer groups while the previous
    # group attends on a second stream; the same bits as compose + attend
    wl = synth.scaled(L8B, layers=layers, chunks_per_request=3, pool_chunks=3, n_suffix=20)
    _fused_case(wl, host={0, 1, 2})
    _fused_case(synth.scaled(wl, batch=2, chunks_per_request=2, pool_chunks=4), host={1, 3})


@pytest.mark.parametrize("host_chunks", [True, False])
def test_compose_attend_suffix_and_output_in_host_memory(host_chunks):
    # Q, K, V of the suffix, O and lse in pinned host memory: the call copies them through
    # device scratch (per layer group on the pipelined route, around the fused kernel
    # otherwise) and gives the same bits as compose + attend on device buffers
    wl = synth.scaled(L8B, layers=5, chunks_per_request=3, pool_chunks=3, n_suffix=20)
    _fused_case(wl, host={0, 1, 2} if host_chunks else (), host_io=True)


def test_attend_one_layer_and_no_lse_with_host_tensors():
    # c2kv_attend of one layer with its Q, K, V and O in pinned host memory, and
    # c2kv_compose_attend with host tensors and no lse: the same bits as on device buffers
    c2kv = H.lib()
    wl = synth.scaled(L8B, layers=3, chunks_per_request=2, pool_chunks=2, n_suffix=24)
    reqs = synth.requests(wl)
    chunks = H.oracle_chunks_meanpool(wl, [0, 1])
    ctx = H.make_ctx(wl, pool_slots=600, fuse=1)
    try:
        dev = H.load_stored(ctx, wl, chunks)
        q, ks, vs = synth.suffix(wl, layers=3)
        req_ptr = np.cumsum([0] + [len(ids) for ids, _ in reqs])
        flat = [dev[c] for ids, _ in reqs for c in ids]
        offs = [o for _, o_ in reqs for o in o_]
        qd, kd, vd = (H.to_dev(x, wl) for x in (q, ks, vs))
        # reference: all layers on device buffers
        cache = c2kv.c2kv_compose(ctx, req_ptr, flat, offs, suffix_capacity=24)
        ref = torch.empty_like(qd)
        c2kv.c2kv_attend(ctx, cache, -1, qd, kd, vd, 24, ref)
        # layer 1 alone, host buffers
        qh, kh, vh = (x[1:2].cpu().pin_memory() for x in (qd, kd, vd))
        oh = torch.empty(qh.shape, dtype=qh.dtype, pin_memory=True)
        c2kv.c2kv_attend(ctx, cache, 1, qh, kh, vh, 24, oh)
        c2kv.c2kv_sync(ctx)
        assert torch.equal(oh.cuda(), ref[1:2])
        c2kv.c2kv_cache_release(ctx, cache)
        # compose_attend, host buffers, no lse
        qh, kh, vh = (x.cpu().pin_memory() for x in (qd, kd, vd))
        oh = torch.empty(qh.shape, dtype=qh.dtype, pin_memory=True)
        cache = c2kv.c2kv_compose_attend(ctx, req_ptr, flat, offs, 24, qh, kh, vh, 24, oh)
        c2kv.c2kv_sync(ctx)
        assert torch.equal(oh.cuda(), ref)
        c2kv.c2kv_cache_release(ctx, cache)
    finally:
        c2kv.c2kv_destroy(ctx)


def test_compose_attend_refuses_unpinned_host_memory():
    # a CPU tensor the CUDA runtime does not know is refused before anything is launched
    c2kv = H.lib()
    wl = synth.scaled(L8B, layers=1, chunks_per_request=2, pool_chunks=2, n_suffix=8)
    reqs = synth.requests(wl)
    chunks = H.oracle_chunks_meanpool(wl, [0, 1])
    ctx = H.make_ctx(wl, pool_slots=400)
    try:
        dev = H.load_stored(ctx, wl, chunks)
        q, ks, vs = synth.suffix(wl, layers=1)
        qd, kd, vd = (H.to_dev(x, wl) for x in (q, ks, vs))
        out_unpinned = torch.empty(qd.shape, dtype=qd.dtype)          # pageable
        req_ptr = np.cumsum([0] + [len(ids) for ids, _ in reqs])
        flat = [dev[c] for ids, _ in reqs for c in ids]
        offs = [o for _, o_ in reqs for o in o_]
        with pytest.raises(c2kv.C2KVError) as ei:
            c2kv.c2kv_compose_attend(ctx, req_ptr, flat, offs, 8, qd, kd, vd, 8, out_unpinned)
        assert ei.value.status == c2kv.ERR_ARG
        # the context still works
        cache, out, _ = _run(ctx, wl, dev, reqs, q, ks, vs, 8, fused=True)
        assert torch.isfinite(out.float()).all()
        c2kv.c2kv_cache_release(ctx, cache)
    finally:
        c2kv.c2kv_destroy(ctx)


def test_fused_bounds_check_reports_and_recovers():
    c2kv = H.lib()
    wl = synth.scaled(L8B, layers=1, chunks_per_request=2, pool_chunks=2, n_suffix=8)
    reqs = synth.requests(wl)
    chunks = H.oracle_chunks_meanpool(wl, [0, 1])
    ctx = H.make_ctx(wl, pool_slots=400)
    try:
        dev = H.load_stored(ctx, wl, chunks)
        q, ks, vs = synth.suffix(wl, layers=1)
        c2kv.c2kv_inject_fault(ctx, 1)       # the first occurrence points past the pool
        try:
            _run(ctx, wl, dev, reqs, q, ks, vs, 8, fused=True)
        except c2kv.C2KVError as e:
            assert e.status == c2kv.ERR_DEVICE_BOUNDS
        else:
            raise AssertionError("the refused pool row was not reported")
        # the context still works
        cache, out, _ = _run(ctx, wl, dev, reqs, q, ks, vs, 8, fused=True)
        assert torch.isfinite(out.float()).all()
        c2kv.c2kv_cache_release(ctx, cache)
    finally:
        c2kv.c2kv_destroy(ctx)


def test_decode_after_fused_matches_unfused():
    # the cache the fused call leaves behind serves decode exactly as compose + attend's
    c2kv = H.lib()
    wl = synth.scaled(L8B, layers=2, chunks_per_request=4, pool_chunks=4, n_suffix=24)
    reqs = synth.requests(wl)
    chunks = H.oracle_chunks_meanpool(wl, sorted({c for ids, _ in reqs for c in ids}))
    ctx = H.make_ctx(wl, pool_slots=1024)
    try:
        dev = H.load_stored(ctx, wl, chunks)
        q, ks, vs = synth.suffix(wl, layers=2)
        B = len(reqs)
        req_ptr = np.cumsum([0] + [len(ids) for ids, _ in reqs])
        flat = [dev[c] for ids, _ in reqs for c in ids]
        offs = [o for _, o_ in reqs for o in o_]
        qd, kd, vd = (H.to_dev(x, wl) for x in (q, ks, vs))
        out = torch.empty_like(qd)
        gen = torch.Generator(device="cuda").manual_seed(3)
        qn = torch.randn((2, B, wl.n_q_heads, wl.head_dim), device="cuda", generator=gen).bfloat16()
        kn = torch.randn((2, B, wl.n_kv_heads, wl.head_dim), device="cuda", generator=gen).bfloat16()
        vn = torch.randn_like(kn)
        outs = []
        for fused in (True, False):
            if fused:
                cache = c2kv.c2kv_compose_attend(ctx, req_ptr, flat, offs, 32, qd, kd, vd, 24, out)
            else:
                cache = c2kv.c2kv_compose(ctx, req_ptr, flat, offs, suffix_capacity=32)
                c2kv.c2kv_attend(ctx, cache, -1, qd, kd, vd, 24, out)
            od = torch.empty_like(qn)
            c2kv.c2kv_decode(ctx, cache, -1, qn, kn, vn, [24] * B, od)
            c2kv.c2kv_sync(ctx)
            outs.append(od)
            c2kv.c2kv_cache_release(ctx, cache)
        assert torch.equal(outs[0], outs[1])
    finally:
        c2kv.c2kv_destroy(ctx)


@pytest.mark.parametrize("n_suffix,fuse,want_fused", [
    (64, 0, True),        # 64 tokens x 4 heads = 256 query rows: one pair of tiles
    (65, 0, False),       # a second pair: compose, then attend
    (65, 2, True),
    (64, 1, False),
])
def test_fuse_policy(n_suffix, fuse, want_fused):
    c2kv = H.lib()
    wl = synth.scaled(L8B, layers=1, chunks_per_request=2, pool_chunks=2, n_suffix=n_suffix)
    reqs = synth.requests(wl)
    chunks = H.oracle_chunks_meanpool(wl, [0, 1])
    ctx = H.make_ctx(wl, pool_slots=400, fuse=fuse)
    try:
        dev = H.load_stored(ctx, wl, chunks)
        q, ks, vs = synth.suffix(wl, layers=1)
        c2kv.c2kv_profile_enable(ctx, True)
        cache, _, _ = _run(ctx, wl, dev, reqs, q, ks, vs, n_suffix, fused=True)
        kinds = c2kv.c2kv_profile_read(ctx)
        assert (kinds["fused"][1] == 1) == want_fused
        assert (kinds["compose"][1] == 1) == (not want_fused)
        c2kv.c2kv_cache_release(ctx, cache)
    finally:
        c2kv.c2kv_destroy(ctx)


def test_fused_traced_and_on_a_side_stream_give_the_same_bits():
    # the fused kernel is launched as the dependent of the suffix-angles kernel: with the
    # library's trace on, events sit between the two, and on another stream the whole call
    # runs there; the cache, O and lse must not change
    c2kv = H.lib()
    wl = synth.scaled(L8B, layers=2, chunks_per_request=3, pool_chunks=3)
    reqs = synth.requests(wl)
    chunks = H.oracle_chunks_meanpool(wl, [0, 1, 2])
    ctx = H.make_ctx(wl, pool_slots=600, fuse=2)
    try:
        dev = H.load_stored(ctx, wl, chunks)
        q, ks, vs = synth.suffix(wl, layers=2)
        runs = [_run(ctx, wl, dev, reqs, q, ks, vs, wl.n_suffix, fused=True)]
        c2kv.c2kv_profile_enable(ctx, True)
        runs.append(_run(ctx, wl, dev, reqs, q, ks, vs, wl.n_suffix, fused=True))
        assert c2kv.c2kv_profile_read(ctx)["fused"][1] == 1
        c2kv.c2kv_profile_enable(ctx, False)
        side = torch.cuda.Stream()
        with torch.cuda.stream(side):
            c2kv.c2kv_set_stream(ctx, side)
            runs.append(_run(ctx, wl, dev, reqs, q, ks, vs, wl.n_suffix, fused=True))
        torch.cuda.synchronize()
        c2kv.c2kv_set_stream(ctx, torch.cuda.current_stream())
        ref = H.cache_arrays(runs[0][0], wl)
        for cache, out, lse in runs[1:]:
            got = H.cache_arrays(cache, wl)
            for r in range(len(reqs)):
                base, s = ref[0]["row_base"][r], ref[0]["n_slots"][r]
                end = base + (s + wl.n_suffix + 127) // 128 * 128
                assert np.array_equal(got[3][base:s + base + wl.n_suffix], ref[3][base:s + base + wl.n_suffix])
                assert np.array_equal(got[1][:, base:end], ref[1][:, base:end])
                assert np.array_equal(got[2][:, base:end], ref[2][:, base:end])
            assert torch.equal(out, runs[0][1])
            assert torch.equal(lse, runs[0][2])
        for cache, _, _ in runs:
            c2kv.c2kv_cache_release(ctx, cache)
    finally:
        c2kv.c2kv_destroy(ctx)


@pytest.mark.parametrize("n_req,per_req", [(300, 1), (130, 4)])
def test_compose_attend_many_requests_or_occurrences(n_req, per_req):
    # more requests (32) or occurrences (128) than the fused launch takes, even forced: the
    # call composes, then attends in groups of 256 requests; sampled requests against the
    # oracle
    c2kv = H.lib()
    wl = synth.scaled(L8B, layers=1, chunk_tokens=64, ratio_k=4, pool_chunks=5, n_suffix=3,
                      batch=n_req)
    chunks = H.oracle_chunks_meanpool(wl, list(range(5)))
    ctx = H.make_ctx(wl, pool_slots=200, fuse=2)
    try:
        dev = H.load_stored(ctx, wl, chunks)
        rng = np.random.default_rng(5)
        reqs = []
        for _ in range(n_req):
            ids = [int(x) for x in rng.integers(0, 5, per_req)]
            reqs.append((ids, [64 * i for i in range(per_req)]))
        q, ks, vs = synth.suffix(wl, layers=1)
        cache, out, lse = _run(ctx, wl, dev, reqs, q, ks, vs, 3, fused=True)
        got = out.double().cpu().numpy()
        for r in (0, 1, n_req // 2, n_req - 1):
            ids, offs = reqs[r]
            ref = orc.run_request(chunks, ids, offs, q[:, r], ks[:, r], vs[:, r], wl.rope_theta,
                                  wl.dtype)
            H.check_attention(got[:, r], ref["out"], wl, f"O req {r}")
        c2kv.c2kv_cache_release(ctx, cache)
    finally:
        c2kv.c2kv_destroy(ctx)


def test_compose_attend_arg_checks():
    c2kv = H.lib()
    wl = synth.scaled(L8B, layers=1, chunks_per_request=1, pool_chunks=1, n_suffix=4)
    chunks = H.oracle_chunks_meanpool(wl, [0])
    ctx = H.make_ctx(wl, pool_slots=200)
    try:
        dev = H.load_stored(ctx, wl, chunks)
        q = torch.zeros((1, 1, 4, wl.n_q_heads, wl.head_dim), device="cuda", dtype=torch.bfloat16)
        kv = torch.zeros((1, 1, 4, wl.n_kv_heads, wl.head_dim), device="cuda", dtype=torch.bfloat16)
        out = torch.empty_like(q)

        def status(*a):
            try:
                c2kv.c2kv_compose_attend(ctx, *a)
            except c2kv.C2KVError as e:
                return e.status
            return c2kv.OK
        assert status([0, 1], [dev[0]], [0], 4, q, kv, kv, 5, out) == c2kv.ERR_ARG      # n_suffix > capacity
        assert status([0, 1], [dev[0]], [0], 4, None, kv, kv, 4, out) == c2kv.ERR_ARG
        assert status([0, 1], [99], [0], 4, q, kv, kv, 4, out) == c2kv.ERR_BAD_CHUNK
        assert status([0, 1], [dev[0]], [-1], 4, q, kv, kv, 4, out) == c2kv.ERR_POSITIONS
        assert status([0, 1], [dev[0]], [0], 4, q.data_ptr() + 2, kv, kv, 4, out) == c2kv.ERR_ARG
        cache = c2kv.c2kv_compose_attend(ctx, [0, 1], [dev[0]], [0], 4, q, kv, kv, 4, out)
        c2kv.c2kv_sync(ctx)
        c2kv.c2kv_cache_release(ctx, cache)
    finally:
        c2kv.c2kv_destroy(ctx)


def test_unfused_route_suffix_beside_compose():
    # fuse NEVER, no trace: compose on the context's stream while the suffix kernel runs on
    # its second stream, then attention; against the oracle and compose + attend
    _fused_case(synth.scaled(synth.workload("batched"), batch=3, chunks_per_request=4,
                             pool_chunks=32, n_suffix=40), fuse=1)


def test_unfused_route_traced_equals_untraced():
    # with the trace on, the unfused route runs compose, suffix and attention in turn on one
    # stream; without it the suffix kernel runs beside compose: the same bits either way
    c2kv = H.lib()
    wl = synth.scaled(synth.workload("batched"), batch=4, chunks_per_request=3, pool_chunks=8,
                      n_suffix=72, layers=2)
    reqs = synth.requests(wl)
    all_ids = sorted({c for ids, _ in reqs for c in ids})
    chunks = H.oracle_chunks_meanpool(wl, all_ids)
    pool = sum(chunks[c][0].shape[1] for c in all_ids) + 16
    ctx = H.make_ctx(wl, pool_slots=pool, fuse=1)
    try:
        dev = H.load_stored(ctx, wl, chunks)
        q, ks, vs = synth.suffix(wl, layers=wl.layers)
        sq = wl.n_suffix
        runs = []
        for traced in (False, True):
            c2kv.c2kv_profile_enable(ctx, traced)
            cache, out, lse = _run(ctx, wl, dev, reqs, q, ks, vs, sq, fused=True)
            runs.append((H.cache_arrays(cache, wl), out, lse))
            c2kv.c2kv_cache_release(ctx, cache)
        c2kv.c2kv_profile_enable(ctx, False)
        kinds = c2kv.c2kv_profile_read(ctx)
        assert kinds.get("suffix", (0, 0))[1] >= 1 and kinds.get("compose", (0, 0))[1] >= 1
        (info_a, ka, va, pa), out_a, lse_a = runs[0]
        (info_b, kb, vb, pb), out_b, lse_b = runs[1]
        for r in range(len(reqs)):
            base, s = info_a["row_base"][r], info_a["n_slots"][r]
            assert info_b["row_base"][r] == base and info_b["n_slots"][r] == s
            end = base + (s + sq + 127) // 128 * 128
            assert np.array_equal(pa[base:base + s + sq], pb[base:base + s + sq])
            assert np.array_equal(ka[:, base:end], kb[:, base:end])
            assert np.array_equal(va[:, base:end], vb[:, base:end])
        assert torch.equal(out_a, out_b)
        assert torch.equal(lse_a, lse_b)
    finally:
        c2kv.c2kv_destroy(ctx)


@pytest.mark.parametrize("n_req,per_req,want_fused", [
    (32, 4, True),        # 32 requests, 128 occurrences: the fused launch's limits
    (33, 3, False),       # one request more than it takes
    (16, 9, False),       # 144 occurrences
])
def test_fused_route_limits(n_req, per_req, want_fused):
    # forced fusion on one pair of query tiles per (layer, request, KV head): the fused launch
    # takes at most 32 requests and 128 occurrences (its parameter block is kept small),
    # larger calls compose, then attend; either way sampled requests match the oracle
    c2kv = H.lib()
    wl = synth.scaled(L8B, layers=1, chunk_tokens=64, ratio_k=4, pool_chunks=5, n_suffix=3,
                      batch=n_req)
    chunks = H.oracle_chunks_meanpool(wl, list(range(5)))
    ctx = H.make_ctx(wl, pool_slots=200, fuse=2)
    try:
        dev = H.load_stored(ctx, wl, chunks)
        rng = np.random.default_rng(11)
        reqs = [([int(x) for x in rng.integers(0, 5, per_req)], [64 * i for i in range(per_req)])
                for _ in range(n_req)]
        q, ks, vs = synth.suffix(wl, layers=1)
        c2kv.c2kv_profile_enable(ctx, True)
        cache, out, _ = _run(ctx, wl, dev, reqs, q, ks, vs, 3, fused=True)
        kinds = c2kv.c2kv_profile_read(ctx)
        assert (kinds["fused"][1] == 1) == want_fused
        assert (kinds["compose"][1] >= 1) == (not want_fused)
        got = out.double().cpu().numpy()
        for r in (0, n_req - 1):
            ids, offs = reqs[r]
            ref = orc.run_request(chunks, ids, offs, q[:, r], ks[:, r], vs[:, r], wl.rope_theta,
                                  wl.dtype)
            H.check_attention(got[:, r], ref["out"], wl, f"O req {r}")
        c2kv.c2kv_cache_release(ctx, cache)
    finally:
        c2kv.c2kv_destroy(ctx)
