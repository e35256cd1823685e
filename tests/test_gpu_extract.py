"""SIF-masked extraction attention (c2kv_extract_attention) against the oracle."""
import numpy as np
import pytest
import torch

import synth
from oracle import c2kv_oracle as orc
from tests import _gpu_helpers as H

pytestmark = pytest.mark.gpu

L8B = synth.workload("llama8b")
TINY = synth.workload("tiny_f32")


def _extract_case(wl, n, k, layers=1, chunk_id=0, attn_pairs=0):
    c2kv = H.lib()
    wl = synth.scaled(wl, layers=layers)
    q, kk, v = synth.extraction_inputs(wl, chunk_id, n, k)
    ctx = H.make_ctx(wl, pool_slots=64, attn_pairs=attn_pairs)
    try:
        qd, kd, vd = (H.to_dev(x, wl) for x in (q, kk, v))
        out = torch.full_like(qd, float("nan"))
        lse = torch.full((layers, wl.n_q_heads, q.shape[1]), float("nan"), device="cuda")
        c2kv.c2kv_extract_attention(ctx, layers, qd, kd, vd, n, k, out, lse)
        c2kv.c2kv_sync(ctx)
        ref, ref_lse = orc.sif_attention(q, kk, v, n, k, wl.rope_theta, wl.dtype)
        got = out.double().cpu().numpy()
        H.check_attention(got[:, :n], ref[:, :n], wl, "document rows")
        H.check_attention(got[:, n:], ref[:, n:], wl, "C2 rows")
        gl = lse.double().cpu().numpy()
        bad = np.abs(gl - ref_lse) > 1e-3 + 1e-4 * np.abs(ref_lse) + _lse_rounding_bound(q, kk, n, k, wl)
        if bad.any():
            i = np.unravel_index(np.argmax(np.abs(gl - ref_lse)), gl.shape)
            raise AssertionError(f"lse: {bad.sum()} off; worst at {i}: got {gl[i]} want {ref_lse[i]}")
    finally:
        c2kv.c2kv_destroy(ctx)


def _lse_rounding_bound(q, kk, n, k, wl):
    """Per (layer, head, row) bound on the lse difference that storage rounding alone can
    make: both sides store the rotated Q and K in the context dtype but round from different
    rotations (fp32 here, fp64 in the oracle), so an element may differ by one unit in the
    last place (relative 2^-8 for bf16, 2^-24 for fp32).  A score then moves by at most
    rel * sum_c |q_c k_c| / sqrt(d), and lse = log sum exp is 1-Lipschitz in the scores, so
    its change is at most the largest such move over the row's visible keys."""
    rel = 2.0 ** -8 if wl.dtype == "bf16" else 2.0 ** -24
    pos = orc.sif_positions(n, k)
    vis = orc.sif_mask(n, k)
    layers, n_all, hq, d = q.shape
    grp = hq // kk.shape[2]
    out = np.zeros((layers, hq, n_all))
    for layer in range(layers):
        q_r = np.abs(orc.store(orc.rope(q[layer], pos, wl.rope_theta), wl.dtype))
        k_r = np.abs(orc.store(orc.rope(kk[layer], pos, wl.rope_theta), wl.dtype))
        for h in range(hq):
            mag = q_r[:, h, :] @ k_r[:, h // grp, :].T / np.sqrt(d)
            out[layer, h] = rel * np.where(vis, mag, 0.0).max(axis=1)
    return out


@pytest.mark.parametrize("n,k", [(512, 4), (77, 4), (203, 10), (64, 1), (40, 64), (1030, 4),
                                 (1999, 16), (1, 1), (5, 3)])
def test_extract_bf16(n, k):
    _extract_case(L8B, n, k)


@pytest.mark.parametrize("hq,hkv", [(8, 8), (16, 8), (32, 2)])
def test_extract_bf16_group_sizes(hq, hkv):
    # G = 1, 2 and 16 query heads per KV head (one to sixteen tokens per 128-row tile)
    _extract_case(synth.scaled(L8B, n_q_heads=hq, n_kv_heads=hkv), 333, 4)


def test_extract_without_lse_matches_with_lse():
    # without an lse array the C2 rows' partial normaliser goes to library scratch; the
    # outputs are the same bits either way
    c2kv = H.lib()
    wl = synth.scaled(L8B, layers=2)
    n, k = 700, 4
    q, kk, v = synth.extraction_inputs(wl, 5, n, k)
    ctx = H.make_ctx(wl, pool_slots=64)
    try:
        qd, kd, vd = (H.to_dev(x, wl) for x in (q, kk, v))
        a = torch.full_like(qd, float("nan"))
        b = torch.full_like(qd, float("nan"))
        lse = torch.empty((2, wl.n_q_heads, q.shape[1]), device="cuda")
        c2kv.c2kv_extract_attention(ctx, 2, qd, kd, vd, n, k, a, lse)
        c2kv.c2kv_extract_attention(ctx, 2, qd, kd, vd, n, k, b)
        c2kv.c2kv_sync(ctx)
        assert torch.equal(a, b)
        ref, _ = orc.sif_attention(q, kk, v, n, k, wl.rope_theta, wl.dtype)
        H.check_attention(b.double().cpu().numpy(), ref, wl, "no-lse call")
    finally:
        c2kv.c2kv_destroy(ctx)


@pytest.mark.parametrize("per_cta", [2, 3, 8])
def test_extract_pairs_run_in_turn(per_cta):
    # the attention launches of the call with several pairs of query tiles per CTA (the
    # document rows have 8 pairs of 1 to 4 key tiles at n = 512): 3 leaves a group of two
    _extract_case(L8B, 512, 4, layers=1, attn_pairs=per_cta)


def test_extract_two_layers_gqa8():
    _extract_case(synth.workload("long70b"), 300, 16, layers=2)


def test_extract_f32_tiny():
    _extract_case(TINY, 128, 4, layers=1)


def test_extract_document_rows_equal_suffix_free_prefill():
    # original-token invariance on the device: perturbing every C2 token leaves the document
    # rows bit-identical
    c2kv = H.lib()
    wl = synth.scaled(L8B, layers=1)
    n, k = 96, 8
    q, kk, v = synth.extraction_inputs(wl, 3, n, k)
    ctx = H.make_ctx(wl, pool_slots=64)
    try:
        outs = []
        for bump in (0.0, 1.0):
            k2, v2, q2 = kk.copy(), v.copy(), q.copy()
            k2[:, n:] += bump
            v2[:, n:] -= bump
            q2[:, n:] *= 1.0 + bump
            qd, kd, vd = (H.to_dev(x, wl) for x in (q2, k2, v2))
            out = torch.empty_like(qd)
            c2kv.c2kv_extract_attention(ctx, 1, qd, kd, vd, n, k, out)
            c2kv.c2kv_sync(ctx)
            outs.append(out[:, :n].clone())
        assert torch.equal(outs[0], outs[1])
    finally:
        c2kv.c2kv_destroy(ctx)
