"""PRE_ROPE storage (c2kv_config.storage = C2KV_STORAGE_PRE_ROPE) against the oracle.

Sec. 3.3.1 stores the C2 tokens' KV before positional embeddings are applied.  Under this
setting the pool keeps K before RoPE and compose applies RoPE at the composed position
o_i + p_j once (oracle: ``compose_pre_rope``, then the storage rounding), where the default
LOCAL_ROPE setting stores K turned to p_j and turns it by o_i.

Tolerances: positions and V bit-exact; composed K one storage ulp of the fp64 result (or
2^-20 of the pair's magnitude where the pair nearly cancels); attention 2e-2 / 1e-5."""
import numpy as np
import pytest
import torch

import synth
from oracle import c2kv_oracle as orc
from tests import _gpu_helpers as H

pytestmark = pytest.mark.gpu

L8B_1 = synth.scaled(synth.workload("llama8b"), layers=1)
TINY = synth.workload("tiny_f32")


def _pre_slots(wl, ids):
    """Pre-RoPE stored slots per chunk id: the synthetic stand-ins for what a storage tier
    holds (exact in the storage dtype), in the oracle's chunk format."""
    m = orc.n_slots(wl.chunk_tokens, wl.ratio_k)
    out = {}
    for cid in ids:
        kb, vb = synth.chunk_slots(wl, cid, m)
        out[cid] = (kb.astype(np.float64), vb.astype(np.float64), wl.chunk_tokens, wl.ratio_k)
    return out


def _load(ctx, wl, slots, host=(), keep=None):
    c2kv = H.lib()
    ids = {}
    for cid, (kb, vb, n, k) in slots.items():
        if cid in host:
            kh, vh = (torch.from_numpy(x.astype(np.float32)).to(H.tdtype(wl)).pin_memory()
                      for x in (kb, vb))
            keep.extend((kh, vh))
            ids[cid] = c2kv.c2kv_compress_chunk(ctx, kh, vh, n, k, c2kv.MODE_HOST)
        else:
            ids[cid] = c2kv.c2kv_compress_chunk(ctx, H.to_dev(kb, wl), H.to_dev(vb, wl), n, k,
                                                c2kv.MODE_STORED)
    return ids


def _expected(wl, slots, ids, offs, fixed_pos=False):
    """(K' fp64 unrounded, V, positions, L_req) of one request composed from pre-RoPE slots."""
    l_req = orc.check_positions([slots[c][2] for c in ids], offs)
    turn_offs = [0] * len(offs) if fixed_pos else list(offs)
    k, v, pos = orc.compose_pre_rope(slots, ids, turn_offs, wl.rope_theta)
    return k, v, pos, l_req


def _compose_case(wl, reqs, fixed_pos=False, host=()):
    c2kv = H.lib()
    all_ids = sorted({c for ids, _ in reqs for c in ids})
    slots = _pre_slots(wl, all_ids)
    pool = sum(s[0].shape[1] for s in slots.values()) + 16
    ctx = H.make_ctx(wl, pool_slots=pool, fixed_pos=int(fixed_pos), storage=c2kv.STORAGE_PRE_ROPE)
    keep = []
    try:
        dev = _load(ctx, wl, slots, host=host, keep=keep)
        req_ptr = np.cumsum([0] + [len(ids) for ids, _ in reqs])
        cache = c2kv.c2kv_compose(ctx, req_ptr, [dev[c] for ids, _ in reqs for c in ids],
                                  [o for _, offs in reqs for o in offs], 8)
        c2kv.c2kv_sync(ctx)
        info, gk, gv, gpos = H.cache_arrays(cache, wl)
        for r, (ids, offs) in enumerate(reqs):
            if not ids:
                continue
            ek, ev, epos, l_req = _expected(wl, slots, ids, offs, fixed_pos)
            base, s = info["row_base"][r], info["n_slots"][r]
            assert s == ek.shape[1] and info["l_req"][r] == l_req
            assert np.array_equal(gpos[base:base + s], epos)
            assert np.array_equal(gv[:, base:base + s], ev)
            pre = np.concatenate([slots[c][0] for c in ids], axis=1)
            H.check_rotated(gk[:, base:base + s], ek, pre, wl, f"PRE_ROPE compose K req {r}")
        c2kv.c2kv_cache_release(ctx, cache)
    finally:
        c2kv.c2kv_destroy(ctx)


def test_pre_rope_compose_llama8b_layer():
    _compose_case(L8B_1, synth.requests(L8B_1))


def test_pre_rope_compose_tiny_f32():
    _compose_case(TINY, synth.requests(TINY))


def test_pre_rope_compose_ragged_gaps_duplicates_two_layers():
    wl = synth.scaled(L8B_1, layers=2, chunk_tokens=203, ratio_k=10, pool_chunks=5)
    reqs = [([0, 3, 0], [7, 300, 800]), ([4], [0]), ([], []), ([2, 1, 4, 3], [0, 203, 406, 10000])]
    _compose_case(wl, reqs)


def test_pre_rope_compose_fixed_pos_and_host_chunks():
    wl = synth.scaled(L8B_1, layers=2, chunk_tokens=203, ratio_k=10, pool_chunks=5)
    reqs = [([0, 3, 0], [7, 300, 800]), ([2, 1, 4, 3], [0, 203, 406, 10000])]
    _compose_case(wl, reqs, fixed_pos=True)
    _compose_case(wl, reqs, host={0, 2, 4})


def test_pre_rope_compose_130_occurrences_one_launch():
    # more occurrences than one compose launch held before (96): one launch now
    wl = synth.scaled(L8B_1, chunk_tokens=64, ratio_k=4, pool_chunks=40)
    rng = np.random.default_rng(5)
    reqs = []
    for r in range(13):
        ids = [int(i) for i in rng.choice(40, size=10, replace=True)]
        reqs.append((ids, [64 * i + 3 * r for i in range(10)]))
    _compose_case(wl, reqs)


def test_pre_rope_meanpool_compress_keeps_k_before_rope():
    c2kv = H.lib()
    wl = synth.scaled(L8B_1, layers=2, chunk_tokens=77, ratio_k=4)
    ctx = H.make_ctx(wl, pool_slots=256, storage=c2kv.STORAGE_PRE_ROPE)
    try:
        kt, vt = synth.chunk_tokens(wl, 0)
        dev = c2kv.c2kv_compress_chunk(ctx, H.to_dev(kt, wl), H.to_dev(vt, wl), 77, 4,
                                       c2kv.MODE_MEANPOOL)
        c2kv.c2kv_sync(ctx)
        gk, gv = H.pool_rows(ctx, wl, dev, 256)
        want_k = orc.store(orc.meanpool_slots(kt, 4), wl.dtype)
        want_v = orc.store(orc.meanpool_slots(vt, 4), wl.dtype)
        H.check_rounded(gk, want_k, orc.meanpool_slots(np.abs(kt.astype(np.float64)), 4), wl, "K")
        H.check_rounded(gv, want_v, orc.meanpool_slots(np.abs(vt.astype(np.float64)), 4), wl, "V")
    finally:
        c2kv.c2kv_destroy(ctx)


@pytest.mark.parametrize("wl", [synth.scaled(L8B_1, layers=2, chunks_per_request=3, pool_chunks=3,
                                             n_suffix=40), TINY], ids=["bf16", "f32"])
def test_pre_rope_compose_attend_matches_oracle(wl):
    # the fused kernel turns per occurrence; PRE_ROPE turns per slot, so the call composes,
    # then attends (even when fusion is forced)
    c2kv = H.lib()
    reqs = synth.requests(wl)
    all_ids = sorted({c for ids, _ in reqs for c in ids})
    slots = _pre_slots(wl, all_ids)
    pool = sum(s[0].shape[1] for s in slots.values()) + 16
    ctx = H.make_ctx(wl, pool_slots=pool, storage=c2kv.STORAGE_PRE_ROPE, fuse=c2kv.FUSE_ALWAYS)
    try:
        dev = _load(ctx, wl, slots)
        q, ks, vs = synth.suffix(wl)
        qd, kd, vd = (H.to_dev(x, wl) for x in (q, ks, vs))
        out = torch.empty_like(qd)
        req_ptr = np.cumsum([0] + [len(ids) for ids, _ in reqs])
        c2kv.c2kv_profile_enable(ctx, True)
        cache = c2kv.c2kv_compose_attend(ctx, req_ptr, [dev[c] for ids, _ in reqs for c in ids],
                                         [o for _, offs in reqs for o in offs], wl.n_suffix,
                                         qd, kd, vd, wl.n_suffix, out)
        kern = c2kv.c2kv_profile_read(ctx)
        assert kern["fused"][1] == 0 and kern["compose"][1] >= 1
        got = out.double().cpu().numpy()
        for r, (ids, offs) in enumerate(reqs):
            ek, ev, _, l_req = _expected(wl, slots, ids, offs)
            o, _ = orc.attend(orc.store(ek, wl.dtype), ev, l_req, q[:, r], ks[:, r], vs[:, r],
                              wl.rope_theta, wl.dtype)
            H.check_attention(got[:, r], o, wl, f"PRE_ROPE attention req {r}")
        c2kv.c2kv_cache_release(ctx, cache)
    finally:
        c2kv.c2kv_destroy(ctx)


def test_pre_rope_equals_local_rope_within_rounding():
    # the same chunk stored both ways composes to the same cache up to one rounding step:
    # LOCAL_ROPE stores round(RoPE(K, p_j)) and turns that by o_i, PRE_ROPE turns K once
    c2kv = H.lib()
    wl = synth.scaled(L8B_1, chunks_per_request=3, pool_chunks=3)
    reqs = synth.requests(wl)
    slots = _pre_slots(wl, [0, 1, 2])
    outs = []
    for storage in (c2kv.STORAGE_LOCAL_ROPE, c2kv.STORAGE_PRE_ROPE):
        ctx = H.make_ctx(wl, pool_slots=512, storage=storage)
        try:
            ids = {}
            for cid, (kb, vb, n, k) in slots.items():
                ids[cid] = c2kv.c2kv_compress_chunk(ctx, H.to_dev(kb, wl), H.to_dev(vb, wl), n, k,
                                                    c2kv.MODE_PROVIDED)
            (rid, offs), = reqs
            cache = c2kv.c2kv_compose(ctx, [0, len(rid)], [ids[c] for c in rid], offs, 4)
            c2kv.c2kv_sync(ctx)
            outs.append(H.cache_arrays(cache, wl))
            c2kv.c2kv_cache_release(ctx, cache)
        finally:
            c2kv.c2kv_destroy(ctx)
    (_, k_loc, v_loc, p_loc), (_, k_pre, v_pre, p_pre) = outs
    assert np.array_equal(p_loc, p_pre) and np.array_equal(v_loc, v_pre)
    ek, _, _, _ = _expected(wl, slots, *reqs[0])
    s = ek.shape[1]
    pre = np.concatenate([slots[c][0] for c in reqs[0][0]], axis=1)
    H.check_rotated(k_pre[:, :s], ek, pre, wl, "PRE_ROPE")
    # LOCAL_ROPE rounds the stored K (half an ulp of a component, at most 2^-8 of the pair's
    # magnitude M in bf16) and turns that error with the pair, then rounds again: within one
    # ulp of the exact value plus 2^-7 M
    diff = np.abs(k_loc[:, :s] - ek)
    allowed = H.ulp_of(ek, wl) + 2.0 ** -7 * H.pair_magnitude(pre)
    assert (diff <= allowed).all()


def test_storage_setting_refused_when_unknown():
    c2kv = H.lib()
    with pytest.raises(c2kv.C2KVError) as ei:
        H.make_ctx(L8B_1, pool_slots=16, storage=7)
    assert ei.value.status == c2kv.ERR_ARG
