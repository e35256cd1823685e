"""Host-side arithmetic of bench.py that its roofline figures rest on."""
import numpy as np
import pytest

import bench
import synth
from oracle import c2kv_oracle as orc


@pytest.mark.parametrize("n,k", [(512, 4), (77, 4), (203, 10), (64, 1), (40, 64), (1, 1),
                                 (1999, 16), (4096, 16)])
def test_sif_visible_pairs_is_the_mask_count(n, k):
    assert bench.sif_visible_pairs(n, k) == int(orc.sif_mask(n, k).sum())


def test_attention_flops_match_the_mask():
    # 4 d flops per visible (query head, key) pair, counted from the oracle's definition of
    # what a suffix token sees (every composed slot, suffix tokens 0..t)
    wl = synth.workload("llama8b")
    f = bench.workload_facts(wl)
    s, sq = f["slots"], wl.n_suffix
    vis = np.ones((sq, s + sq), dtype=bool)
    vis[:, s:] = np.tril(np.ones((sq, sq), dtype=bool))
    want = 4.0 * wl.head_dim * wl.n_q_heads * vis.sum() * wl.batch * wl.layers
    assert f["attn_flops"] == pytest.approx(want)


def test_fused_step_reports_compose_and_attention_rooflines():
    # the fused kernel carries "roofline"; the separate compose and attention kernels of the
    # unfused steps are reported beside it, each against the HBM peak here
    f = {"compose_bytes": 335544320, "attn_flops": 44040192000, "attn_bytes": 209715200,
         "name": "llama8b", "fused_bytes": 385881088}
    r = bench.step_rooflines(True, {"fused": (0.0926, 1)}, 0.0606, 0.0585, f, 6790.3, 1904.5, "measured")
    assert r["roofline"]["kernel"].startswith("attn_tc_kernel<fused>")
    assert r["roofline_compose"]["kernel"] == "compose_bulk_kernel"
    assert abs(r["roofline_compose"]["frac"] - 335544320 / 0.0606e-3 / 6790.3e9) < 1e-3
    assert r["roofline_attend"]["kernel"] == "attn_tc_kernel"
    unfused = bench.step_rooflines(False, {}, 0.0606, 0.0585, f, 6790.3, 1904.5, "measured")
    assert {o["kernel"] for o in unfused.values()} == {"compose_bulk_kernel", "attn_tc_kernel"}


def test_compose_bytes_count_every_slot_once():
    # read and write of K and V per composed slot and layer, plus one int32 position per
    # slot, with the slot count from the oracle's definition of m = ceil(n / k)
    for name in ("llama8b", "long70b", "sweep_k10", "tiny_f32"):
        wl = synth.workload(name)
        f = bench.workload_facts(wl)
        m = orc.n_slots(wl.chunk_tokens, wl.ratio_k)
        slots = wl.batch * wl.chunks_per_request * m
        eb = 4 if wl.dtype == "f32" else 2
        want = 2 * 2 * slots * wl.n_kv_heads * wl.head_dim * eb * wl.layers + 4 * slots
        assert f["compose_bytes"] == want, name


@pytest.mark.parametrize("name,keys,tc", [("llama8b", 1360, False), ("sweep_k1", 32907, True),
                                          ("batched", 1163, True), ("long70b", 2315, True),
                                          ("tiny_f32", 160, False)])
def test_decode_line_names_the_route_kernel(name, keys, tc):
    # the library's rule: bf16 at head_dim 128 on the tensor cores when the (layer, request,
    # KV head) units fit in one wave of SMs or a request has 32 key tiles or more
    wl = synth.workload(name)
    line = bench.decode_line(wl, 1, 0.05, 0.04, keys * wl.batch, 6790.3, "measured")
    kernel = line["roofline"]["kernel"]
    assert kernel.startswith("attn_tc_decode_kernel" if tc else "decode_kernel"), kernel
    # algorithmic bytes: K and V of every key, every layer and KV head, once
    eb = 4 if wl.dtype == "f32" else 2
    assert line["roofline"]["bytes_per_launch"] == keys * wl.batch * wl.layers * wl.n_kv_heads * wl.head_dim * eb * 2


def test_reference_arm_line_matches_the_contract():
    # the oracle arm: one JSON line with impl "reference", the GPU arm's metric, unit and
    # config object, its own cpu_baseline and an e2e object with no host-device bytes
    import json
    import os
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    res = subprocess.run([sys.executable, os.path.join(root, "bench.py"), "--impl", "reference",
                          "--steps", "3", "--warmup", "3"], capture_output=True, text=True,
                         timeout=300, cwd=root)
    assert res.returncode == 0, res.stderr[-2000:]
    line = json.loads(res.stdout.strip().splitlines()[-1])
    assert line["impl"] == "reference"
    assert line["metric"] == "composed KV tokens/s" and line["unit"] == "tokens/s"
    assert line["higher_is_better"] is True and line["steps"] == 3 and line["warmup"] == 3
    assert line["config"] == bench.job_config(synth.workload("llama8b"), 1)
    assert line["value"] > 0 and line["ms_per_step"] > 0
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["value"] == line["value"]
    assert line["e2e"] == {"value": line["value"], "unit": line["unit"],
                           "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}
