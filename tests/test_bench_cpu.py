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
