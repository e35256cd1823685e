"""Full-size parity: every workload at its real size, run the way bench.py runs it (one
c2kv_compose_attend call for all layers and requests: on llama8b the fused compose +
attention kernel, elsewhere one compose launch and one attend with layer = -1), checked
against the oracle on sampled outputs (chosen layers / requests, all of their rows).

llama8b and tiny_f32 run the whole chain from tokens (GPU mean-pool compress -> compose
-> attend) against the oracle's chain; the larger pools load random stored slots (the
storage-tier form) to keep input generation short.
"""
import numpy as np
import pytest
import torch

import synth
from oracle import c2kv_oracle as orc
from tests import _gpu_helpers as H

pytestmark = pytest.mark.gpu


def _run_full(wl, from_tokens, sample_layers, sample_reqs, seed=0, fuse=0):
    c2kv = H.lib()
    reqs = synth.requests(wl, seed)
    pool_ids = sorted({c for ids, _ in reqs for c in ids})
    m = orc.n_slots(wl.chunk_tokens, wl.ratio_k)
    ctx = H.make_ctx(wl, pool_slots=len(pool_ids) * m + 8, fuse=fuse)
    needed = {c for r in sample_reqs for c in reqs[r][0]}
    oracle_chunks = {}
    v_scale = {}        # block mean of |v|: the operand scale of the fp32 mean
    try:
        dev = {}
        for cid in pool_ids:
            if from_tokens:
                kt, vt = synth.chunk_tokens(wl, cid, seed)
                dev[cid] = c2kv.c2kv_compress_chunk(ctx, H.to_dev(kt, wl), H.to_dev(vt, wl),
                                                    wl.chunk_tokens, wl.ratio_k,
                                                    c2kv.MODE_MEANPOOL)
                if cid in needed:
                    ks, vs = orc.compress_chunk(kt[sample_layers], vt[sample_layers],
                                                wl.chunk_tokens, wl.ratio_k, wl.rope_theta,
                                                wl.dtype, "meanpool")
                    oracle_chunks[cid] = (ks, vs, wl.chunk_tokens, wl.ratio_k)
                    v_scale[cid] = orc.meanpool_slots(np.abs(vt[sample_layers].astype(np.float64)),
                                                      wl.ratio_k)
            else:
                ks, vs = synth.chunk_slots(wl, cid, m, seed)
                dev[cid] = c2kv.c2kv_compress_chunk(ctx, H.to_dev(ks, wl), H.to_dev(vs, wl),
                                                    wl.chunk_tokens, wl.ratio_k,
                                                    c2kv.MODE_STORED)
                if cid in needed:
                    oracle_chunks[cid] = (ks[sample_layers].astype(np.float64),
                                          vs[sample_layers].astype(np.float64),
                                          wl.chunk_tokens, wl.ratio_k)
            torch.cuda.current_stream().synchronize()
        req_ptr = np.cumsum([0] + [len(ids) for ids, _ in reqs])
        q, ks_, vs_ = synth.suffix(wl, seed)
        qd, kd, vd = (H.to_dev(x, wl) for x in (q, ks_, vs_))
        out = torch.full_like(qd, float("nan"))
        cache = c2kv.c2kv_compose_attend(ctx, req_ptr, [dev[c] for ids, _ in reqs for c in ids],
                                         [o for _, offs in reqs for o in offs], wl.n_suffix,
                                         qd, kd, vd, wl.n_suffix, out)
        c2kv.c2kv_sync(ctx)
        info = c2kv.c2kv_cache_info(cache)
        shp = (info["layers"], info["rows"], wl.n_kv_heads, wl.head_dim)
        k_all = c2kv.device_view(info["k"], shp, H.tdtype(wl))
        v_all = c2kv.device_view(info["v"], shp, H.tdtype(wl))
        pos = c2kv.device_view(info["pos"], (info["rows"],), torch.int32).cpu().numpy()
        for r in sample_reqs:
            ids, offs = reqs[r]
            ref = orc.run_request(oracle_chunks, ids, offs, q[sample_layers, r],
                                  ks_[sample_layers, r], vs_[sample_layers, r],
                                  wl.rope_theta, wl.dtype)
            base, s = int(info["row_base"][r]), int(info["n_slots"][r])
            assert np.array_equal(pos[base:base + s], ref["pos"])
            gv = v_all[sample_layers, base:base + s].double().cpu().numpy()
            gk = k_all[sample_layers, base:base + s].double().cpu().numpy()
            if from_tokens:
                # the GPU compressed its own copy: V within one ulp of the oracle's mean
                # (or fp32 sum error relative to the block's inputs)
                scale = np.concatenate([v_scale[c] for c in ids], axis=1)
                H.check_rounded(gv, ref["v"], scale, wl, f"{wl.name} V req {r}")
                # composed K: the oracle's compose of the slots the GPU stored (the compress
                # step is checked above through V and below through O) within one ulp
                pool = len(pool_ids) * m + 8
                gpu_chunks = {}
                for c in set(ids):
                    pk, pv = H.pool_rows(ctx, wl, dev[c], pool)
                    gpu_chunks[c] = (pk[sample_layers], pv[sample_layers], wl.chunk_tokens, wl.ratio_k)
                ck, _, _, _ = orc.compose(gpu_chunks, ids, offs, wl.rope_theta, wl.dtype)
                stored = np.concatenate([gpu_chunks[c][0] for c in ids], axis=1)
                H.check_rotated(gk, ck, stored, wl, f"{wl.name} K req {r}")
            else:
                assert np.array_equal(gv, ref["v"])
                stored = np.concatenate([oracle_chunks[c][0] for c in ids], axis=1)
                H.check_rotated(gk, ref["k"], stored, wl, f"{wl.name} K req {r}")
            got = out[sample_layers, r].double().cpu().numpy()
            H.check_attention(got, ref["out"], wl, f"{wl.name} O req {r}")
        assert torch.isfinite(out.float()).all()
        c2kv.c2kv_cache_release(ctx, cache)
    finally:
        c2kv.c2kv_destroy(ctx)


def test_full_tiny_f32():
    _run_full(synth.workload("tiny_f32"), True, [0], [0])


def test_full_llama8b_32_layers():
    _run_full(synth.workload("llama8b"), True, [0, 13, 31], [0])            # fused


def test_full_llama8b_32_layers_unfused():
    _run_full(synth.workload("llama8b"), True, [0, 13, 31], [0], fuse=1)   # compose, attend


def test_full_batched_zipf():
    _run_full(synth.workload("batched"), False, [0], [0, 7, 15])


def test_full_batched_zipf_fused():
    # the fused kernel forced on 16 requests with two query-tile pairs each
    _run_full(synth.workload("batched"), False, [0], [0, 7, 15], fuse=2)


def test_full_long70b_fused():
    # the fused kernel forced where every key tile holds two occurrences (64 slots each)
    _run_full(synth.workload("long70b"), False, [0], [0, 1], fuse=2)


def test_full_long70b():
    _run_full(synth.workload("long70b"), False, [0], [0, 1])


@pytest.mark.parametrize("k", synth.SWEEP_RATIOS)
def test_full_sweep(k):
    _run_full(synth.workload(f"sweep_k{k}"), False, [0], [0, 7])
