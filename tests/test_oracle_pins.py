"""Pins for the CPU oracle: each check ties an oracle function to something other than
itself (a value the paper prints, a textbook formulation, a library routine, brute
force, or an exact identity).  Checks take the implementation as an argument so the
mutation tests at the bottom can plant a mistake in a copy of the oracle and show
that some pin fails."""
import math
import os

import numpy as np
import pytest
import torch

from oracle import c2kv_oracle as orc

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
RNG = np.random.default_rng(1234)


# ------------------------------------------------------------------ storage rounding

def test_round_to_bf16_ties_and_values():
    r = orc.round_to_bf16
    # 1 + 2^-8 is halfway between 1 and 1 + 2^-7: ties to even -> 1.
    assert r(np.array([1 + 2.0**-8]))[0] == 1.0
    # 1 + 3*2^-8 is halfway between 1+2^-7 (odd) and 1+2^-6 (even) -> 1+2^-6.
    assert r(np.array([1 + 3 * 2.0**-8]))[0] == 1 + 2.0**-6
    assert r(np.array([-3.0]))[0] == -3.0
    assert r(np.array([0.0]))[0] == 0.0
    # just above a tie rounds up
    assert r(np.array([1 + 2.0**-8 + 2.0**-30]))[0] == 1 + 2.0**-7


def test_round_to_bf16_matches_torch_on_f32_inputs():
    # For inputs that are already float32, one rounding from fp64 equals torch's
    # float32 -> bfloat16 conversion (round to nearest even).
    x = (RNG.standard_normal(20000) * np.exp(RNG.uniform(-20, 20, 20000))).astype(np.float32)
    want = torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy()
    got = orc.round_to_bf16(x.astype(np.float64))
    assert np.array_equal(got, want)


# ------------------------------------------------------------------ slots and positions

def _golden_positions():
    rows = []
    for line in open(os.path.join(GOLDEN, "slot_positions.txt")):
        if not line.strip() or line.startswith("#"):
            continue
        lhs, rhs = line.split("|")
        n, k = map(int, lhs.split())
        rows.append((n, k, [int(t) for t in rhs.split()]))
    return rows


def check_slot_positions_golden(slot_pos_fn, n_slots_fn):
    for n, k, want in _golden_positions():
        if list(slot_pos_fn(n, k)) != want or n_slots_fn(n, k) != len(want):
            return False
    return True


def _walk_blocks(n, k):
    """Brute force: stream the tokens one by one, closing a block every k tokens or at
    the end of the chunk, and note the index of the token that closes it."""
    closers, count = [], 0
    for t in range(n):
        count += 1
        if count == k or t == n - 1:
            closers.append(t)
            count = 0
    return closers


def check_slot_positions_bruteforce(slot_pos_fn, n_slots_fn):
    for n in range(0, 65):
        for k in (1, 2, 3, 4, 8, 10, 16):
            want = _walk_blocks(n, k)
            if n_slots_fn(n, k) != len(want) or list(slot_pos_fn(n, k)) != want:
                return False
    return True


def test_slot_positions_golden():
    assert check_slot_positions_golden(orc.slot_local_positions, orc.n_slots)


def test_slot_positions_bruteforce():
    assert check_slot_positions_bruteforce(orc.slot_local_positions, orc.n_slots)


def test_compression_ratio_golden_parse():
    lines = [ln.split() for ln in open(os.path.join(GOLDEN, "compression_ratios.txt"))
             if ln.strip() and not ln.startswith("#")]
    table = {ln[0]: [int(v) for v in ln[1:]] for ln in lines}
    assert table["dynamic_test"] == [4, 8, 10, 16] and table["default"] == [4]
    # the sweep workload uses exactly these plus the uncompressed control
    import synth
    assert list(synth.SWEEP_RATIOS) == [1] + table["dynamic_test"]


# ------------------------------------------------------------------ RoPE

def rope_complex(x, pos, theta):
    """Textbook RoPE as complex multiplication: z_i = x_i + i x_{i+d/2}, z_i * e^{i p w_i}
    with w_i = theta^(-2i/d) computed as exp(-2i/d * ln theta)."""
    x = np.asarray(x, np.float64)
    d = x.shape[-1]
    w = np.exp(-(2.0 * np.arange(d // 2) / d) * math.log(theta))
    z = x[..., : d // 2] + 1j * x[..., d // 2:]
    rot = np.exp(1j * np.outer(np.asarray(pos, np.float64), w))[:, None, :]
    zr = z * rot
    return np.concatenate([zr.real, zr.imag], axis=-1)


def check_rope_textbook(rope_fn):
    x = RNG.standard_normal((37, 3, 16))
    pos = RNG.integers(0, 40000, 37)
    for theta in (1e4, 5e5):
        if not np.allclose(rope_fn(x, pos, theta), rope_complex(x, pos, theta),
                           rtol=1e-9, atol=1e-9):
            return False
    return True


def check_rope_hand_values(rope_fn):
    # d = 4, theta = 1e4: frequencies (1, 0.01).  Channel 0 pairs with 2, 1 with 3.
    x = np.zeros((2, 1, 4))
    x[0, 0, 0] = 1.0                 # turns by 1 rad/position
    x[1, 0, 1] = 1.0                 # turns by 0.01 rad/position
    out = rope_fn(x, np.array([2, 100]), 1e4)
    want0 = [math.cos(2.0), 0.0, math.sin(2.0), 0.0]
    want1 = [0.0, math.cos(1.0), 0.0, math.sin(1.0)]
    return np.allclose(out[0, 0], want0, atol=1e-14) and np.allclose(out[1, 0], want1,
                                                                      atol=1e-12)


def test_rope_textbook():
    assert check_rope_textbook(orc.rope)


def test_rope_hand_values():
    assert check_rope_hand_values(orc.rope)


def test_rope_group_and_inverse():
    # North-star identities: turning by D then -D is the identity; K cached at p and
    # turned by D equals K computed at p + D (1e-6 relative required; ~1e-12 in fp64).
    x = RNG.standard_normal((64, 8, 128))
    p = RNG.integers(0, 4096, 64)
    for delta in (1, 17, 4096, 32767):
        dl = np.full(64, delta)
        back = orc.rope(orc.rope(x, dl, 5e5), -dl, 5e5)
        assert np.max(np.abs(back - x)) < 1e-12
        shifted = orc.rope(orc.rope(x, p, 5e5), dl, 5e5)
        direct = orc.rope(x, p + delta, 5e5)
        rel = np.max(np.abs(shifted - direct)) / np.max(np.abs(direct))
        assert rel < 1e-6 and rel < 1e-11


def test_rope_preserves_pair_norms_and_relative_scores():
    x = RNG.standard_normal((10, 2, 64))
    y = orc.rope(x, np.arange(10) * 977, 1e4)
    nx = x[..., :32] ** 2 + x[..., 32:] ** 2
    ny = y[..., :32] ** 2 + y[..., 32:] ** 2
    assert np.allclose(nx, ny, rtol=1e-12)
    # <RoPE(q, a), RoPE(k, b)> depends only on a - b
    q = RNG.standard_normal((1, 1, 64))
    k = RNG.standard_normal((1, 1, 64))
    s1 = np.sum(orc.rope(q, [500], 1e4) * orc.rope(k, [123], 1e4))
    s2 = np.sum(orc.rope(q, [500 + 9000], 1e4) * orc.rope(k, [123 + 9000], 1e4))
    assert abs(s1 - s2) < 1e-10


# ------------------------------------------------------------------ mean pooling

def meanpool_loops(tok, k):
    """Brute force block means with explicit loops (tok [n, H, d])."""
    n, h, d = tok.shape
    out = []
    start = 0
    while start < n:
        end = min(start + k, n)
        row = np.zeros((h, d))
        for t in range(start, end):
            row += tok[t]
        out.append(row / (end - start))
        start = end
    return np.array(out)


def check_meanpool_bruteforce(meanpool_fn):
    for n in (1, 3, 9, 16, 21):
        for k in (1, 2, 3, 4, 10):
            tok = RNG.standard_normal((n, 2, 4))
            if not np.allclose(meanpool_fn(tok[None], k)[0], meanpool_loops(tok, k),
                               rtol=1e-13, atol=1e-13):
                return False
    return True


def test_meanpool_bruteforce():
    assert check_meanpool_bruteforce(orc.meanpool_slots)


def test_meanpool_special_cases():
    tok = RNG.standard_normal((1, 12, 2, 8))
    assert np.array_equal(orc.meanpool_slots(tok, 1), tok)           # k = 1 is identity
    const = np.repeat(RNG.standard_normal((1, 1, 2, 8)), 12, axis=1)
    assert np.allclose(orc.meanpool_slots(const, 5), const[:, :3])    # constant rows


def test_compress_k1_is_plain_prefill_cache():
    # k = 1, mean pooling: every slot is its own token, stored at its own position;
    # this is the uncompressed control, bit-exact round trip of V.
    k_tok = orc.round_to_bf16(RNG.standard_normal((2, 9, 2, 8)))
    v_tok = orc.round_to_bf16(RNG.standard_normal((2, 9, 2, 8)))
    k_st, v_st = orc.compress_chunk(k_tok, v_tok, 9, 1, 1e4, "bf16", "meanpool")
    assert np.array_equal(v_st, v_tok)
    for layer in range(2):
        want = orc.round_to_bf16(rope_complex(k_tok[layer], np.arange(9), 1e4))
        assert np.array_equal(k_st[layer], want)


# ------------------------------------------------------------------ composition

def _random_chunks(lengths, ks, L=2, H=2, d=8, theta=1e4):
    """Pre-RoPE slot values and their locally-rotated stored form (fp64, unrounded)."""
    pre, stored = {}, {}
    for cid, (n, k) in enumerate(zip(lengths, ks)):
        m = orc.n_slots(n, k)
        kb = RNG.standard_normal((L, m, H, d))
        vb = RNG.standard_normal((L, m, H, d))
        pre[cid] = (kb, vb, n, k)
        ks_, vs_ = orc.compress_chunk(kb, vb, n, k, theta, "f64", "provided")
        stored[cid] = (ks_, vs_, n, k)
    return pre, stored


def test_compose_local_rope_equals_pre_rope():
    lengths, ks = [9, 16, 7, 30], [4, 4, 10, 16]
    pre, stored = _random_chunks(lengths, ks)
    ids = [2, 0, 3, 1, 0]
    positions = [5, 20, 29, 70, 200]
    k_c, v_c, pos, l_req = orc.compose(stored, ids, positions, 1e4, "f64")
    k_p, v_p, pos_p = orc.compose_pre_rope(pre, ids, positions, 1e4)
    assert np.max(np.abs(k_c - k_p)) < 1e-12
    assert np.array_equal(v_c, v_p) and np.array_equal(pos, pos_p)
    assert l_req == 200 + 9


def test_compose_positions_bruteforce():
    lengths, ks = [10, 5, 16], [4, 16, 3]
    _, stored = _random_chunks(lengths, ks)
    ids, positions = [1, 2, 0], [3, 8, 40]
    _, _, pos, l_req = orc.compose(stored, ids, positions, 1e4, "f64")
    want = []
    for cid, o in zip(ids, positions):
        want += [o + t for t in _walk_blocks(lengths[cid], ks[cid])]
    assert list(pos) == want and l_req == 50


def test_compose_single_chunk_k1_offset0_is_prefill_cache():
    n, L, H, d = 24, 2, 2, 8
    k_tok = RNG.standard_normal((L, n, H, d))
    v_tok = RNG.standard_normal((L, n, H, d))
    k_st, v_st = orc.compress_chunk(k_tok, v_tok, n, 1, 5e5, "f64", "meanpool")
    k_c, v_c, pos, _ = orc.compose({7: (k_st, v_st, n, 1)}, [7], [0], 5e5, "f64")
    for layer in range(L):
        assert np.allclose(k_c[layer], rope_complex(k_tok[layer], np.arange(n), 5e5),
                           atol=1e-12)
    assert np.array_equal(v_c, v_tok) and list(pos) == list(range(n))


def test_compose_shift_equals_direct_encoding():
    # A chunk encoded at 0..n-1 and composed at offset o equals the same chunk encoded
    # directly at o..o+n-1 (k = 1), to 1e-6 relative (fp64 gives ~1e-12).
    n, o = 16, 12345
    k_tok = RNG.standard_normal((1, n, 2, 16))
    k_st, v_st = orc.compress_chunk(k_tok, k_tok, n, 1, 5e5, "f64", "meanpool")
    k_c, _, pos, _ = orc.compose({0: (k_st, v_st, n, 1)}, [0], [o], 5e5, "f64")
    direct = rope_complex(k_tok[0], o + np.arange(n), 5e5)
    assert np.max(np.abs(k_c[0] - direct)) / np.max(np.abs(direct)) < 1e-11
    assert list(pos) == list(range(o, o + n))


def test_compose_fixed_pos_keeps_local_positions():
    _, stored = _random_chunks([8, 8], [4, 4])
    k_c, v_c, pos, l_req = orc.compose(stored, [0, 1], [0, 8], 1e4, "f64", fixed_pos=True)
    assert np.array_equal(k_c, np.concatenate([stored[0][0], stored[1][0]], axis=1))
    assert list(pos) == [3, 7, 3, 7] and l_req == 16


@pytest.mark.parametrize("bad", [[0, 5], [-1, 20], [20, 0]])
def test_compose_rejects_overlap(bad):
    _, stored = _random_chunks([10, 10], [4, 4])
    with pytest.raises(ValueError):
        orc.compose(stored, [0, 1], bad, 1e4, "f64")


# ------------------------------------------------------------------ attention

def _sdpa_reference(keys, vals, q_r, s_len):
    """torch SDPA in fp64 with an explicit boolean mask and torch's own GQA mapping."""
    sq, hq, d = q_r.shape
    qt = torch.from_numpy(q_r).permute(1, 0, 2)[None]                 # [1, Hq, Sq, d]
    kt = torch.from_numpy(keys).permute(1, 0, 2)[None]
    vt = torch.from_numpy(vals).permute(1, 0, 2)[None]
    t = torch.arange(sq)[:, None]
    j = torch.arange(keys.shape[0])[None, :]
    mask = j <= s_len + t
    o = torch.nn.functional.scaled_dot_product_attention(
        qt, kt, vt, attn_mask=mask, enable_gqa=True)
    return o[0].permute(1, 0, 2).numpy()


def check_attend_vs_sdpa(attend_fn, hq=4, hkv=2):
    """One chunk, k = 1, offset 0: the suffix rows of plain causal attention over
    [chunk; suffix] (computed by torch SDPA) must equal the oracle's output."""
    n, sq, d, theta = 13, 6, 16, 1e4
    k_tok = RNG.standard_normal((1, n, hkv, d))
    v_tok = RNG.standard_normal((1, n, hkv, d))
    q = RNG.standard_normal((1, sq, hq, d))
    k_s = RNG.standard_normal((1, sq, hkv, d))
    v_s = RNG.standard_normal((1, sq, hkv, d))
    k_st, v_st = orc.compress_chunk(k_tok, v_tok, n, 1, theta, "f64", "meanpool")
    k_c, v_c, _, l_req = orc.compose({0: (k_st, v_st, n, 1)}, [0], [0], theta, "f64")
    out, _ = attend_fn(k_c, v_c, l_req, q, k_s, v_s, theta, "f64")
    # full-sequence reference built independently with the complex RoPE
    allk = np.concatenate([k_tok[0], k_s[0]])
    allv = np.concatenate([v_tok[0], v_s[0]])
    keys = rope_complex(allk, np.arange(n + sq), theta)
    q_r = rope_complex(q[0], n + np.arange(sq), theta)
    ref = _sdpa_reference(keys, allv, q_r, n)
    return np.allclose(out[0], ref, rtol=1e-10, atol=1e-12)


def test_attend_vs_sdpa_gqa():
    assert check_attend_vs_sdpa(orc.attend, hq=8, hkv=2)


def test_attend_vs_sdpa_mha():
    assert check_attend_vs_sdpa(orc.attend, hq=3, hkv=3)


def test_attend_bruteforce_loops():
    # Tiny case by explicit loops: S = 3 composed slots, 2 suffix tokens, d = 4.
    s_len, sq, d = 3, 2, 4
    k_c = RNG.standard_normal((1, s_len, 1, d))
    v_c = RNG.standard_normal((1, s_len, 1, d))
    q = RNG.standard_normal((1, sq, 2, d))
    k_s = RNG.standard_normal((1, sq, 1, d))
    v_s = RNG.standard_normal((1, sq, 1, d))
    l_req = 40
    out, lse = orc.attend(k_c, v_c, l_req, q, k_s, v_s, 1e4, "f64")
    for t in range(sq):
        p = l_req + t
        qr = rope_complex(q[0, t:t + 1], [p], 1e4)[0]
        keys = [k_c[0, j, 0] for j in range(s_len)]
        vals = [v_c[0, j, 0] for j in range(s_len)]
        for u in range(t + 1):
            keys.append(rope_complex(k_s[0, u:u + 1], [l_req + u], 1e4)[0, 0])
            vals.append(v_s[0, u, 0])
        for h in range(2):
            sc = [sum(qr[h, c] * kk[c] for c in range(d)) / 2.0 for kk in keys]
            mx = max(sc)
            w = [math.exp(s - mx) for s in sc]
            tot = sum(w)
            o = sum(wi * vv for wi, vv in zip(w, vals)) / tot
            assert np.allclose(out[0, t, h], o, atol=1e-13)
            assert abs(lse[0, h, t] - (mx + math.log(tot))) < 1e-13


def test_attend_slot_permutation_invariance():
    s_len, sq, d = 20, 5, 8
    k_c = RNG.standard_normal((1, s_len, 2, d))
    v_c = RNG.standard_normal((1, s_len, 2, d))
    q = RNG.standard_normal((1, sq, 4, d))
    k_s = RNG.standard_normal((1, sq, 2, d))
    v_s = RNG.standard_normal((1, sq, 2, d))
    perm = RNG.permutation(s_len)
    a, la = orc.attend(k_c, v_c, 100, q, k_s, v_s, 1e4, "f64")
    b, lb = orc.attend(k_c[:, perm], v_c[:, perm], 100, q, k_s, v_s, 1e4, "f64")
    assert np.allclose(a, b, atol=1e-13) and np.allclose(la, lb, atol=1e-13)


def _decode_case(s_len, step, hq=4, hkv=2, d=8, l_req=70):
    k_c = RNG.standard_normal((2, s_len, hkv, d))
    v_c = RNG.standard_normal((2, s_len, hkv, d))
    q = RNG.standard_normal((2, step + 1, hq, d))
    k_s = RNG.standard_normal((2, step + 1, hkv, d))
    v_s = RNG.standard_normal((2, step + 1, hkv, d))
    return k_c, v_c, q, k_s, v_s, l_req


@pytest.mark.parametrize("s_len,step", [(20, 0), (20, 4), (0, 3), (33, 9)])
def test_decode_step_equals_last_row_of_attend(s_len, step):
    # one query over every key vs the masked matrix form: row `step` of a suffix of
    # step + 1 tokens sees exactly the keys the decode step sees
    k_c, v_c, q, k_s, v_s, l_req = _decode_case(s_len, step)
    out, lse = orc.decode_step(k_c, v_c, l_req, k_s[:, :step], v_s[:, :step], q[:, step],
                               k_s[:, step], v_s[:, step], step, 1e4, "f64")
    full, lse_full = orc.attend(k_c, v_c, l_req, q, k_s, v_s, 1e4, "f64")
    assert np.allclose(out, full[:, step], atol=1e-13)
    assert np.allclose(lse, lse_full[:, :, step], atol=1e-13)


def test_decode_step_closed_forms():
    d = 8
    empty = np.zeros((1, 0, 1, d))
    # a single key: the output is its value and the lse is the scaled score
    q = RNG.standard_normal((1, 2, d))
    k = RNG.standard_normal((1, 1, d))
    v = RNG.standard_normal((1, 1, d))
    out, lse = orc.decode_step(empty, empty, 5, empty, empty, q, k, v, 0, 1e4, "f64")
    assert np.allclose(out[0, 0], v[0, 0], atol=1e-15) and np.allclose(out[0, 1], v[0, 0], atol=1e-15)
    qr = rope_complex(q[0][None], [5], 1e4)[0]                 # [Hq, d]
    kr = rope_complex(k[0][None], [5], 1e4)[0, 0]              # [d]
    assert abs(lse[0, 0] - qr[0] @ kr / math.sqrt(d)) < 1e-12
    assert abs(lse[0, 1] - qr[1] @ kr / math.sqrt(d)) < 1e-12
    # all keys zero (a rotated zero stays zero): every score is 0, the weights are uniform
    # over the 6 composed slots and the new token, and lse = log 7
    vals = RNG.standard_normal((1, 6, 1, d))
    v_new = RNG.standard_normal((1, 1, d))
    out, lse = orc.decode_step(np.zeros((1, 6, 1, d)), vals, 9, empty, empty, q[:, :1],
                               np.zeros((1, 1, d)), v_new, 0, 1e4, "f64")
    mean = (vals[0, :, 0].sum(axis=0) + v_new[0, 0]) / 7.0
    assert np.allclose(out[0, 0], mean, atol=1e-14)
    assert abs(lse[0, 0] - math.log(7.0)) < 1e-13


def _sif_case(n, k, hq=4, hkv=2, d=8, layers=1):
    m = orc.n_slots(n, k)
    q = RNG.standard_normal((layers, n + m, hq, d))
    kk = RNG.standard_normal((layers, n + m, hkv, d))
    v = RNG.standard_normal((layers, n + m, hkv, d))
    return q, kk, v


@pytest.mark.parametrize("n,k", [(13, 4), (8, 8), (9, 1), (20, 30)])
def test_sif_document_rows_are_causal_attention(n, k):
    # original-token invariance: the document rows equal plain causal attention over the
    # document alone (torch SDPA in fp64, its own causal mask and GQA mapping)
    q, kk, v = _sif_case(n, k)
    out, _ = orc.sif_attention(q, kk, v, n, k, 1e4, "f64")
    q_r = rope_complex(q[0, :n], np.arange(n), 1e4)
    k_r = rope_complex(kk[0, :n], np.arange(n), 1e4)
    qt = torch.from_numpy(q_r).permute(1, 0, 2)[None]
    kt = torch.from_numpy(k_r).permute(1, 0, 2)[None]
    vt = torch.from_numpy(v[0, :n]).permute(1, 0, 2)[None]
    ref = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, is_causal=True,
                                                           enable_gqa=True)
    assert np.allclose(out[0, :n], ref[0].permute(1, 0, 2).numpy(), atol=1e-12)


def test_sif_c2_rows_bruteforce():
    # C2 token c_j by explicit loops over the key set the paper states: B(j), the first
    # block (sink), and c_0 .. c_j; positions are block ends
    n, k, d = 10, 4, 4
    q, kk, v = _sif_case(n, k, hq=2, hkv=1, d=d)
    out, lse = orc.sif_attention(q, kk, v, n, k, 1e4, "f64")
    m = orc.n_slots(n, k)
    for j in range(m):
        end = min((j + 1) * k, n)
        keys = sorted(set(range(j * k, end)) | set(range(0, min(k, n))) |
                      {n + i for i in range(j + 1)})
        def posof(t):
            return t if t < n else min((t - n + 1) * k, n) - 1
        qr = rope_complex(q[0, n + j][None], [posof(n + j)], 1e4)[0]
        for h in range(2):
            sc = []
            for u in keys:
                kr = rope_complex(kk[0, u][None], [posof(u)], 1e4)[0, 0]
                sc.append(sum(qr[h, c] * kr[c] for c in range(d)) / 2.0)
            mx = max(sc)
            w = [math.exp(x - mx) for x in sc]
            o = sum(wi * v[0, u, 0] for wi, u in zip(w, keys)) / sum(w)
            assert np.allclose(out[0, n + j, h], o, atol=1e-13)
            assert abs(lse[0, h, n + j] - (mx + math.log(sum(w)))) < 1e-13


def test_sif_mask_structure():
    n, k = 11, 3
    vis = orc.sif_mask(n, k)
    m = orc.n_slots(n, k)
    assert not vis[:n, n:].any()                           # documents never see C2 tokens
    assert (vis[:n, :n] == np.tril(np.ones((n, n), bool))).all()
    assert (vis[n:, n:] == np.tril(np.ones((m, m), bool))).all()
    # c_j sees exactly its block and the first block among the document tokens
    for j in range(m):
        want = np.zeros(n, bool)
        want[j * k:min((j + 1) * k, n)] = True
        want[:k] = True
        assert (vis[n + j, :n] == want).all()


def test_pins_catch_a_leaky_sif_mask(monkeypatch):
    # a mask that lets document tokens see the C2 tokens breaks original-token invariance
    good = orc.sif_mask

    def leaky(n, k):
        vis = good(n, k)
        vis[:n, n:] = True
        return vis
    monkeypatch.setattr(orc, "sif_mask", leaky)
    with pytest.raises(AssertionError):
        test_sif_document_rows_are_causal_attention(13, 4)


def test_pins_catch_a_sif_mask_that_sees_ahead(monkeypatch):
    # c_j also seeing c_{j+1} (a causal accumulation shifted by one) fails the brute force
    good = orc.sif_mask

    def ahead(n, k):
        vis = good(n, k)
        m = vis.shape[0] - n
        for j in range(m - 1):
            vis[n + j, n + j + 1] = True
        return vis
    monkeypatch.setattr(orc, "sif_mask", ahead)
    with pytest.raises(AssertionError):
        test_sif_c2_rows_bruteforce()


def test_pins_catch_a_sif_sink_taken_as_the_last_block(monkeypatch):
    # reading the sink block as the chunk's last block instead of its first fails the pins
    good = orc.sif_mask

    def last_sink(n, k):
        vis = good(n, k)
        m = vis.shape[0] - n
        for j in range(m):
            vis[n + j, :n] = False
            vis[n + j, j * k:min((j + 1) * k, n)] = True
            vis[n + j, (m - 1) * k:n] = True
        return vis
    monkeypatch.setattr(orc, "sif_mask", last_sink)
    with pytest.raises(AssertionError):
        test_sif_c2_rows_bruteforce()


def test_lse_combine_equals_unsplit():
    s_len, sq, d, hq, hkv = 50, 7, 8, 4, 2
    keys = RNG.standard_normal((s_len + sq, hkv, d))
    vals = RNG.standard_normal((s_len + sq, hkv, d))
    q_r = RNG.standard_normal((sq, hq, d))
    vis = np.arange(s_len + sq)[None, :] <= (s_len + np.arange(sq))[:, None]
    full, lse_full = orc.attend_partial(keys, vals, q_r, vis)
    cuts = [0, 17, 40, s_len + sq]
    outs, lses = [], []
    for a, b in zip(cuts[:-1], cuts[1:]):
        o, l_ = orc.attend_partial(keys[a:b], vals[a:b], q_r, vis[:, a:b])
        outs.append(o)
        lses.append(l_)
    got, lse = orc.lse_combine(outs, lses)
    assert np.allclose(got, full, atol=1e-13) and np.allclose(lse, lse_full, atol=1e-13)


# ------------------------------------------------------------------ planted mistakes

def test_pins_catch_planted_rope_mistakes():
    def wrong_sign(x, pos, theta):
        return orc.rope(x, -np.asarray(pos), theta)

    def adjacent_pairs(x, pos, theta):        # interleaved pairing instead of rotate-half
        x = np.asarray(x, np.float64)
        d = x.shape[-1]
        y = np.empty_like(x)
        y[..., : d // 2], y[..., d // 2:] = x[..., 0::2], x[..., 1::2]
        r = orc.rope(y, pos, theta)
        out = np.empty_like(r)
        out[..., 0::2], out[..., 1::2] = r[..., : d // 2], r[..., d // 2:]
        return out

    def wrong_freq(x, pos, theta):            # theta^(-i/d) instead of theta^(-2i/d)
        return orc.rope(x, pos, math.sqrt(theta))

    for bad in (wrong_sign, adjacent_pairs, wrong_freq):
        assert not (check_rope_textbook(bad) and check_rope_hand_values(bad))


def test_pins_catch_planted_slot_and_pool_mistakes():
    def first_token(n, k):                    # position of the first token instead
        return np.array([j * k for j in range(orc.n_slots(n, k))])

    def floor_count(n, k):
        return n // k

    assert not check_slot_positions_bruteforce(first_token, orc.n_slots)
    assert not check_slot_positions_golden(orc.slot_local_positions, floor_count)

    def divide_by_k(tok, k):                  # the equation's 1/k on a partial block
        n = tok.shape[-3]
        return np.stack([tok[..., a:b, :, :].sum(axis=-3) / k
                         for a, b in (orc.block(j, n, k) for j in range(orc.n_slots(n, k)))],
                        axis=-3)

    assert not check_meanpool_bruteforce(divide_by_k)


def test_pins_catch_planted_attention_mistakes(monkeypatch):
    def no_causal(k_c, v_c, l_req, q, k_s, v_s, theta, dtype):
        # everything visible: drop the causal mask inside the suffix
        n_layers, s_len, hkv, d = k_c.shape
        sq, hq = q.shape[1], q.shape[2]
        pos = orc.suffix_positions(l_req, sq)
        q_r = orc.rope(q[0], pos, theta)
        keys = np.concatenate([k_c[0], orc.rope(k_s[0], pos, theta)])
        vals = np.concatenate([v_c[0], v_s[0]])
        o, lse = orc.attend_partial(keys, vals, q_r, np.ones((sq, s_len + sq), bool))
        return o[None], lse[None]

    assert not check_attend_vs_sdpa(no_causal, hq=4, hkv=2)

    # GQA mapping h % Hkv instead of h // (Hq/Hkv)
    real_attend = orc.attend

    def modulo_groups(k_c, v_c, l_req, q, k_s, v_s, theta, dtype):
        hq, hkv = q.shape[2], k_c.shape[2]
        order = [(h % hkv) * (hq // hkv) + h // hkv for h in range(hq)]
        inv = np.argsort(order)
        o, lse = real_attend(k_c, v_c, l_req, q[:, :, order], k_s, v_s, theta, dtype)
        return o[:, :, inv], lse[:, inv]

    assert not check_attend_vs_sdpa(modulo_groups, hq=8, hkv=2)

    # scale 1/d instead of 1/sqrt(d)
    monkeypatch.setattr(orc.math, "sqrt", lambda v: v)
    assert not check_attend_vs_sdpa(orc.attend, hq=4, hkv=2)
