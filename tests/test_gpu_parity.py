"""GPU vs oracle parity for the three steps of the path (compress, compose, attend),
all through the C ABI.  Sizes here keep the oracle at seconds while spanning several
128-row tiles and a ragged tail; the full-size cases are in test_gpu_fullsize.py.

Tolerances (stated per check):
  slot positions, composed positions, V copies: bit-exact;
  rotated K: one storage ulp of the fp64 result rounded once, or 2^-20 of the pair's
    magnitude where the pair nearly cancels (fp32 rotation arithmetic);
  attention output: |gpu - oracle| <= tol + tol * |oracle|, tol = 2e-2 (bf16), 1e-5 (fp32).
"""
import numpy as np
import pytest
import torch

import synth
from oracle import c2kv_oracle as orc
from tests import _gpu_helpers as H

pytestmark = pytest.mark.gpu

TINY = synth.workload("tiny_f32")
L8B_1 = synth.scaled(synth.workload("llama8b"), layers=1)


def _small(wl, **kw):
    return synth.scaled(wl, **kw)


# ------------------------------------------------------------------ compress

@pytest.mark.parametrize("wl", [
    TINY,
    _small(L8B_1, layers=2, chunk_tokens=77, ratio_k=4, chunks_per_request=2, pool_chunks=2),
    _small(L8B_1, chunk_tokens=203, ratio_k=10, chunks_per_request=2, pool_chunks=2),
    _small(L8B_1, chunk_tokens=64, ratio_k=1, chunks_per_request=1, pool_chunks=1),
    _small(L8B_1, chunk_tokens=512, ratio_k=16, chunks_per_request=1, pool_chunks=1),
    _small(TINY, n_kv_heads=1, n_q_heads=4, head_dim=128, chunk_tokens=9, ratio_k=4),
], ids=["tiny_f32", "bf16_ragged_k4_2layers", "bf16_k10", "bf16_k1", "bf16_k16",
        "f32_d128_ragged"])
def test_compress_meanpool(wl):
    c2kv = H.lib()
    ctx = H.make_ctx(wl, pool_slots=2048)
    try:
        for cid in range(min(2, wl.pool_chunks)):
            kt, vt = synth.chunk_tokens(wl, cid)
            dev = c2kv.c2kv_compress_chunk(ctx, H.to_dev(kt, wl), H.to_dev(vt, wl),
                                           wl.chunk_tokens, wl.ratio_k, c2kv.MODE_MEANPOOL)
            c2kv.c2kv_sync(ctx)
            info = c2kv.c2kv_chunk_info(ctx, dev)
            assert info["n_slots"] == orc.n_slots(wl.chunk_tokens, wl.ratio_k)
            gk, gv = H.pool_rows(ctx, wl, dev, 2048)
            ok, ov = orc.compress_chunk(kt, vt, wl.chunk_tokens, wl.ratio_k, wl.rope_theta,
                                        wl.dtype, "meanpool")
            # operand scale: block mean of |pair| (K) and of |v| (V); fp32 sums of fp32
            # inputs round relative to the inputs, not to their (possibly small) mean
            k_scale = orc.meanpool_slots(H.pair_magnitude(kt.astype(np.float64)), wl.ratio_k)
            v_scale = orc.meanpool_slots(np.abs(vt.astype(np.float64)), wl.ratio_k)
            H.check_rounded(gk, ok, k_scale, wl, "meanpool K")
            # V: mean only; a copy for k = 1
            if wl.ratio_k == 1:
                assert np.array_equal(gv, ov)
            else:
                H.check_rounded(gv, ov, v_scale, wl, "meanpool V")
    finally:
        c2kv.c2kv_destroy(ctx)


def test_compress_provided():
    wl = _small(L8B_1, layers=2, chunk_tokens=300, ratio_k=8)
    c2kv = H.lib()
    m = orc.n_slots(wl.chunk_tokens, wl.ratio_k)
    kb, vb = synth.chunk_slots(wl, 5, m)
    ctx = H.make_ctx(wl, pool_slots=512)
    try:
        dev = c2kv.c2kv_compress_chunk(ctx, H.to_dev(kb, wl), H.to_dev(vb, wl),
                                       wl.chunk_tokens, wl.ratio_k, c2kv.MODE_PROVIDED)
        gk, gv = H.pool_rows(ctx, wl, dev, 512)
        ok, ov = orc.compress_chunk(kb, vb, wl.chunk_tokens, wl.ratio_k, wl.rope_theta,
                                    wl.dtype, "provided")
        H.check_rotated(gk, ok, kb.astype(np.float64), wl, "provided K")
        assert np.array_equal(gv, ov)
    finally:
        c2kv.c2kv_destroy(ctx)


def test_compress_stored_roundtrip_from_host():
    # STORED from pageable host memory (numpy) and from pinned host memory: verbatim.
    wl = _small(L8B_1, layers=3)
    c2kv = H.lib()
    m = 37
    ks, vs = synth.chunk_slots(wl, 1, m)
    ctx = H.make_ctx(wl, pool_slots=200)
    try:
        kh = torch.from_numpy(ks).to(torch.bfloat16)
        vh = torch.from_numpy(vs).to(torch.bfloat16).pin_memory()
        dev = c2kv.c2kv_compress_chunk(ctx, kh, vh, m * 4, 4, c2kv.MODE_STORED)
        c2kv.c2kv_sync(ctx)
        gk, gv = H.pool_rows(ctx, wl, dev, 200)
        assert np.array_equal(gk, ks.astype(np.float64))
        assert np.array_equal(gv, vs.astype(np.float64))
    finally:
        c2kv.c2kv_destroy(ctx)


# ------------------------------------------------------------------ compose

def _compose_case(wl, requests, fixed_pos=False, pool_slots=4096, host=()):
    """Compose `requests` (list of (ids, offsets)) on the GPU from oracle-stored chunks and
    compare every request with the oracle's compose.  Chunks named in `host` stay in pinned
    host memory (MODE_HOST) and compose reads them there."""
    c2kv = H.lib()
    all_ids = sorted({c for ids, _ in requests for c in ids})
    chunks = H.oracle_chunks_meanpool(wl, all_ids)
    ctx = H.make_ctx(wl, pool_slots=pool_slots, fixed_pos=int(fixed_pos))
    keep = []
    try:
        dev = H.load_stored(ctx, wl, chunks, host=host, keep=keep)
        req_ptr = np.cumsum([0] + [len(ids) for ids, _ in requests])
        flat_ids = [dev[c] for ids, _ in requests for c in ids]
        flat_pos = [o for _, offs in requests for o in offs]
        cache = c2kv.c2kv_compose(ctx, req_ptr, flat_ids, flat_pos, suffix_capacity=8)
        c2kv.c2kv_sync(ctx)
        info, gk, gv, gpos = H.cache_arrays(cache, wl)
        for r, (ids, offs) in enumerate(requests):
            if not ids:                       # a request that reuses no chunk
                assert info["n_slots"][r] == 0 and info["l_req"][r] == 0
                assert info["capacity"][r] == 128
                continue
            ok, ov, opos, l_req = orc.compose(chunks, ids, offs, wl.rope_theta, wl.dtype,
                                              fixed_pos)
            base, s = info["row_base"][r], info["n_slots"][r]
            assert base % 128 == 0
            assert s == ok.shape[1] and info["l_req"][r] == l_req
            assert info["capacity"][r] >= s + 8 and info["capacity"][r] % 128 == 0
            assert np.array_equal(gpos[base:base + s], opos)              # bit-exact
            assert np.array_equal(gv[:, base:base + s], ov)               # bit-exact copy
            stored = np.concatenate([chunks[c][0] for c in ids], axis=1)
            H.check_rotated(gk[:, base:base + s], ok, stored, wl, f"compose K req {r}")
        c2kv.c2kv_cache_release(ctx, cache)
    finally:
        c2kv.c2kv_destroy(ctx)


def test_compose_tiny_f32():
    _compose_case(TINY, synth.requests(TINY))


def test_compose_llama8b_layer():
    _compose_case(L8B_1, synth.requests(L8B_1))


def test_compose_batch_duplicates_gaps_ragged():
    wl = _small(L8B_1, layers=2, chunk_tokens=203, ratio_k=10, pool_chunks=5)
    reqs = [([0, 3, 0], [7, 300, 800]),        # duplicate chunk, gaps (system prompt)
            ([4], [0]),
            ([2, 1, 4, 3], [0, 203, 406, 10000])]
    _compose_case(wl, reqs)


def test_compose_fixed_pos():
    wl = _small(L8B_1, chunks_per_request=3, pool_chunks=3)
    _compose_case(wl, [([0, 1, 2], [0, 512, 1024])], fixed_pos=True)


def test_compose_default_positions_are_prefix_sums():
    c2kv = H.lib()
    wl = _small(L8B_1, chunk_tokens=100, ratio_k=4, pool_chunks=3)
    chunks = H.oracle_chunks_meanpool(wl, [0, 1, 2])
    ctx = H.make_ctx(wl, pool_slots=1024)
    try:
        dev = H.load_stored(ctx, wl, chunks)
        cache = c2kv.c2kv_compose(ctx, [0, 3], [dev[2], dev[0], dev[1]], None, 4)
        info, gk, gv, gpos = H.cache_arrays(cache, wl)
        ok, ov, opos, l_req = orc.compose(chunks, [2, 0, 1], [0, 100, 200], wl.rope_theta,
                                          wl.dtype)
        assert np.array_equal(gpos[:ok.shape[1]], opos) and info["l_req"][0] == 300
    finally:
        c2kv.c2kv_destroy(ctx)


def test_compose_empty_request_in_batch():
    wl = _small(L8B_1, chunk_tokens=64, pool_chunks=2)
    _compose_case(wl, [([0, 1], [0, 64]), ([], []), ([1], [5])])


def test_compose_host_chunks():
    # every chunk stays in pinned host memory: compose reads, re-rotates and gathers it
    # in one pass; V and positions bit-exact as from the pool
    _compose_case(L8B_1, synth.requests(L8B_1), host=set(range(L8B_1.pool_chunks)))


def test_compose_host_and_pool_chunks_mixed():
    wl = _small(L8B_1, layers=2, chunk_tokens=203, ratio_k=10, pool_chunks=5)
    reqs = [([0, 3, 0], [7, 300, 800]),
            ([4], [0]),
            ([2, 1, 4, 3], [0, 203, 406, 10000])]
    _compose_case(wl, reqs, host={0, 2, 4})
    _compose_case(wl, reqs, host={0, 1, 2, 3, 4}, fixed_pos=True)


def test_host_chunks_take_no_pool_slots():
    # a pool of 8 slots composes host chunks of 103 slots each; freeing them leaves the pool
    # untouched (a pool chunk of 8 slots still fits afterwards)
    c2kv = H.lib()
    wl = _small(L8B_1, layers=2, chunk_tokens=412, ratio_k=4, pool_chunks=3)
    chunks = H.oracle_chunks_meanpool(wl, [0, 1, 2])
    ctx = H.make_ctx(wl, pool_slots=8)
    keep = []
    try:
        dev = H.load_stored(ctx, wl, chunks, host={0, 1, 2}, keep=keep)
        info = c2kv.c2kv_chunk_info(ctx, dev[1])
        assert info["n_slots"] == 103 and info["layer_stride"] == 103 * wl.n_kv_heads * wl.head_dim
        cache = c2kv.c2kv_compose(ctx, [0, 3], [dev[2], dev[0], dev[1]], [0, 412, 824], 4)
        info_c, gk, gv, gpos = H.cache_arrays(cache, wl)
        ok, ov, opos, l_req = orc.compose(chunks, [2, 0, 1], [0, 412, 824], wl.rope_theta,
                                          wl.dtype)
        assert np.array_equal(gpos[:ok.shape[1]], opos) and np.array_equal(gv[:, :ok.shape[1]], ov)
        c2kv.c2kv_cache_release(ctx, cache)
        for c in (0, 1, 2):
            c2kv.c2kv_free_chunk(ctx, dev[c])
        ks, vs = synth.chunk_slots(wl, 9, 8)
        c2kv.c2kv_compress_chunk(ctx, H.to_dev(ks, wl), H.to_dev(vs, wl), 32, 4,
                                 c2kv.MODE_STORED)
    finally:
        c2kv.c2kv_destroy(ctx)


def test_host_mode_rejects_pageable_and_misaligned():
    # both refusals are taken on the host before anything is enqueued
    c2kv = H.lib()
    wl = _small(L8B_1, layers=1)
    ctx = H.make_ctx(wl, pool_slots=64)
    try:
        ks, vs = synth.chunk_slots(wl, 1, 8)
        kp = torch.from_numpy(ks).to(torch.bfloat16)                   # pageable
        vp = torch.from_numpy(vs).to(torch.bfloat16)
        with pytest.raises(c2kv.C2KVError) as ei:
            c2kv.c2kv_compress_chunk(ctx, kp, vp, 32, 4, c2kv.MODE_HOST)
        assert ei.value.status == c2kv.ERR_ARG
        buf = torch.zeros(2 * ks.size + 8, dtype=torch.bfloat16).pin_memory()
        with pytest.raises(c2kv.C2KVError) as ei:                      # 2-byte offset
            c2kv.c2kv_compress_chunk(ctx, buf.data_ptr() + 2, buf.data_ptr() + 2 * ks.size + 2,
                                     32, 4, c2kv.MODE_HOST)
        assert ei.value.status == c2kv.ERR_ARG
    finally:
        c2kv.c2kv_destroy(ctx)


# ------------------------------------------------------------------ attend

def _attend_case(wl, attn_impl=0, layer=-1, n_suffix=None, requests=None, attn_split=0,
                 host=()):
    """End to end: oracle-stored chunks -> GPU compose -> GPU attend, vs oracle compose +
    attend on the same inputs.  Checks O, lse, and the suffix rows written to the cache.
    Chunks named in `host` stay in pinned host memory (MODE_HOST)."""
    c2kv = H.lib()
    sq = wl.n_suffix if n_suffix is None else n_suffix
    wl = synth.scaled(wl, n_suffix=sq)
    reqs = synth.requests(wl) if requests is None else requests
    all_ids = sorted({c for ids, _ in reqs for c in ids})
    chunks = H.oracle_chunks_meanpool(wl, all_ids)
    ctx = H.make_ctx(wl, pool_slots=sum(orc.n_slots(wl.chunk_tokens, wl.ratio_k)
                                        for _ in all_ids) + 16, attn_impl=attn_impl,
                       attn_split=attn_split)
    keep = []
    try:
        dev = H.load_stored(ctx, wl, chunks, host=host, keep=keep)
        req_ptr = np.cumsum([0] + [len(ids) for ids, _ in reqs])
        cache = c2kv.c2kv_compose(ctx, req_ptr, [dev[c] for ids, _ in reqs for c in ids],
                                  [o for _, offs in reqs for o in offs], suffix_capacity=sq)
        q, ks, vs = synth.suffix(wl, layers=wl.layers)
        B = len(reqs)
        q, ks, vs = q[:, :B], ks[:, :B], vs[:, :B]
        lsel = slice(None) if layer == -1 else slice(layer, layer + 1)
        qd, kd, vd = (H.to_dev(x[lsel], wl) for x in (q, ks, vs))
        out = torch.full_like(qd, float("nan"))
        lse = torch.full((qd.shape[0], B, wl.n_q_heads, sq), float("nan"), device="cuda")
        c2kv.c2kv_attend(ctx, cache, layer, qd, kd, vd, sq, out, lse)
        c2kv.c2kv_sync(ctx)
        info, gk, gv, gpos = H.cache_arrays(cache, wl)
        got = out.double().cpu().numpy()
        got_lse = lse.double().cpu().numpy()
        for r, (ids, offs) in enumerate(reqs):
            ref = orc.run_request(chunks, ids, offs, q[:, r], ks[:, r], vs[:, r],
                                  wl.rope_theta, wl.dtype)
            ref_o = ref["out"][lsel]
            H.check_attention(got[:, r], ref_o, wl, f"O req {r}")
            assert np.allclose(got_lse[:, r], ref["lse"][lsel], atol=1e-3, rtol=1e-4), "lse"
            base, s = info["row_base"][r], info["n_slots"][r]
            assert np.array_equal(gpos[base + s: base + s + sq],
                                  orc.suffix_positions(ref["l_req"], sq))
            lay = np.arange(wl.layers)[lsel]
            assert np.array_equal(gv[lay, base + s: base + s + sq],
                                  vs[lsel, r].astype(np.float64))
        c2kv.c2kv_cache_release(ctx, cache)
    finally:
        c2kv.c2kv_destroy(ctx)


def test_attend_tiny_f32():
    _attend_case(TINY)


@pytest.mark.parametrize("impl", [1, 0], ids=["simt", "auto"])
def test_attend_llama8b_layer(impl):
    _attend_case(L8B_1, attn_impl=impl)


def test_attend_cuda_cores_large_launch():
    # 4 layers x 8 KV heads x 16 CTAs of 16 query rows: a launch large enough that the
    # CUDA-core kernel keeps 16 rows a CTA (smaller launches take 4); a ragged row count
    wl = _small(L8B_1, layers=4, chunks_per_request=2, pool_chunks=2, n_suffix=61)
    _attend_case(wl, attn_impl=1)


@pytest.mark.parametrize("sq", [1, 7, 33, 100])
def test_attend_ragged_suffix(sq):
    wl = _small(L8B_1, chunks_per_request=3, pool_chunks=3, chunk_tokens=300, ratio_k=10)
    _attend_case(wl, n_suffix=sq)


def test_attend_single_layer_of_many():
    wl = _small(L8B_1, layers=4, chunks_per_request=2, pool_chunks=2, n_suffix=20)
    _attend_case(wl, layer=2)


def test_attend_batched_zipf_reduced():
    wl = _small(synth.workload("batched"), batch=3, chunks_per_request=4, pool_chunks=32,
                n_suffix=40)
    _attend_case(wl)


def test_attend_gqa8_long_reduced():
    wl = _small(synth.workload("long70b"), chunks_per_request=4, pool_chunks=8, n_suffix=48)
    _attend_case(wl)


def test_attend_mha_and_d64():
    wl = _small(L8B_1, n_q_heads=4, n_kv_heads=4, head_dim=64, chunks_per_request=2,
                pool_chunks=2, n_suffix=17)
    _attend_case(wl)


def test_attend_f32_larger():
    wl = _small(TINY, chunk_tokens=333, ratio_k=10, n_suffix=45, n_q_heads=8, n_kv_heads=2)
    _attend_case(wl)


def test_attend_single_chunk_k1_offset0_is_causal_attention():
    # The uncompressed control: one chunk, k = 1, offset 0 -> plain causal attention.
    wl = _small(L8B_1, chunk_tokens=200, ratio_k=1, chunks_per_request=1, pool_chunks=1,
                n_suffix=50)
    _attend_case(wl)


@pytest.mark.parametrize("split", [1, 3, 7])
def test_attend_key_range_splits(split):
    # one short chunk and a long suffix: 3 key tiles, so with 7 splits four are empty, and
    # the last non-empty split sees no visible key for the early suffix rows
    wl = _small(L8B_1, chunks_per_request=1, pool_chunks=1, chunk_tokens=64, ratio_k=4,
                n_suffix=300)
    _attend_case(wl, attn_split=split)


def test_attend_from_host_chunks():
    wl = _small(L8B_1, layers=2)
    _attend_case(wl, host=set(range(wl.pool_chunks)))


def test_attend_forced_split_batched():
    wl = _small(synth.workload("batched"), batch=3, chunks_per_request=4, pool_chunks=32,
                n_suffix=40)
    _attend_case(wl, attn_split=5)


def test_attend_output_at_16_byte_offset_matches():
    # the tensor-core epilogue stores 32 bytes at a time when the output is 32-byte aligned,
    # 16 otherwise: an output starting 16 bytes into a buffer gives the same bits, through
    # the per-row stores (CTAs of four pairs of query tiles) and the staged store of the last
    c2kv = H.lib()
    wl = synth.scaled(L8B_1, layers=2, chunks_per_request=3, pool_chunks=3, n_suffix=200)
    reqs = synth.requests(wl)
    all_ids = sorted({c for ids, _ in reqs for c in ids})
    chunks = H.oracle_chunks_meanpool(wl, all_ids)
    ctx = H.make_ctx(wl, pool_slots=sum(orc.n_slots(wl.chunk_tokens, wl.ratio_k) for _ in all_ids) + 16,
                     attn_pairs=4)
    try:
        dev = H.load_stored(ctx, wl, chunks)
        req_ptr = np.cumsum([0] + [len(ids) for ids, _ in reqs])
        cache = c2kv.c2kv_compose(ctx, req_ptr, [dev[c] for ids, _ in reqs for c in ids],
                                  [o for _, offs in reqs for o in offs], suffix_capacity=200)
        q, ks, vs = synth.suffix(wl, layers=wl.layers)
        qd, kd, vd = (H.to_dev(x[:, :1], wl) for x in (q, ks, vs))
        out = torch.full_like(qd, float("nan"))
        c2kv.c2kv_attend(ctx, cache, -1, qd, kd, vd, 200, out)
        buf = torch.full((out.numel() + 8,), float("nan"), dtype=out.dtype, device="cuda")
        off = buf[8:].view(out.shape)                     # 16 bytes past a 256-byte boundary
        assert off.data_ptr() % 32 == 16
        c2kv.c2kv_attend(ctx, cache, -1, qd, kd, vd, 200, off)
        c2kv.c2kv_sync(ctx)
        assert torch.equal(out, off)
        ref = orc.run_request(chunks, reqs[0][0], reqs[0][1], q[:, 0], ks[:, 0], vs[:, 0],
                              wl.rope_theta, wl.dtype)
        H.check_attention(out.double().cpu().numpy()[:, 0], ref["out"], wl, "O")
        c2kv.c2kv_cache_release(ctx, cache)
    finally:
        c2kv.c2kv_destroy(ctx)
