"""Plain, slow fp64 CPU oracle for C2KV compressed-KV composition and suffix attention.

TEST INFRASTRUCTURE ONLY.  Nothing on the product path imports, calls or links this file:
only the tests, the smoke check and the benchmark's CPU-baseline / reference leg use it.
It shares no code with the CUDA library and imports nothing from it.

What it computes (C2KV, arXiv 2607.17715):

* Compression (Sec. 3.2.1, 3.2.3, 3.3.1).  A chunk of n tokens gets m = ceil(n/k) slots;
  slot j stands for block B(j) of k consecutive tokens and takes the position of the last
  token of that block.  The paper's slots come from a trained extractor whose weights are
  not available, so two stand-ins are offered: ``provided`` (the caller passes the m slot
  K/V it obtained elsewhere) and ``meanpool`` (slot = mean of the block's pre-RoPE K/V
  rows, the block mean that the residual mean-pooling variant of Sec. 3.2.3 adds to the
  C2 hidden state).  Stored K carries RoPE at the slot's chunk-local position.
* Composition (Sec. 3.2.4; Appendix C, TTFT protocol).  Slots of the requested chunks are given new
  positional embeddings for their placement (offsets accumulate, each compressed segment
  spans its original token length), then concatenated.  With RoPE this is a rotation of
  the stored K by the chunk's offset; V is copied.
* Inference (Sec. 2.2, Eq. for F).  The suffix (query) tokens run standard attention over
  [composed cache; suffix], causal inside the suffix, every composed slot visible.  A
  decode step is the same operator for one new token over everything cached before it.
* Extraction attention (Sec. 3.3).  The extractor's attention layer over a chunk's
  document tokens and its C2 tokens under the Structured Information Flow mask.

RoPE is the rotate-half form used by the Llama / Qwen models the paper evaluates
(Sec. 4.1): channel i pairs with i + d/2 and turns by pos * theta^(-2i/d).

Readings where the paper is silent (each also listed in the design notes):
  partial last block divides by its true size |B(j)|; composed slot position is
  offset + local position; positions must be non-decreasing and non-overlapping;
  query head h uses KV head h // (Hq/Hkv); stored values are rounded to the storage
  dtype (bf16 round-to-nearest-even, or fp32) each time they are stored.

Every function works in float64 on numpy arrays.
"""
from __future__ import annotations

import math

import numpy as np

# --------------------------------------------------------------------------------------
# Storage rounding
# --------------------------------------------------------------------------------------


def round_to_bf16(x):
    """Round float64 values to the nearest bfloat16 (8 significant bits, ties to even),
    returned as float64.  A single rounding straight from float64."""
    x = np.asarray(x, dtype=np.float64)
    out = np.zeros_like(x)
    nz = (x != 0) & np.isfinite(x)
    _, e = np.frexp(x[nz])                       # x = f * 2**e, 0.5 <= |f| < 1
    q = np.maximum(e - 8, -133).astype(np.float64)  # bf16 quantum (subnormals bottom out)
    scaled = x[nz] * np.exp2(-q)                  # exact: power-of-two scaling
    out[nz] = np.round(scaled) * np.exp2(q)       # np.round is ties-to-even
    out[~nz] = x[~nz]
    return out


def round_to_f32(x):
    return np.asarray(x, dtype=np.float64).astype(np.float32).astype(np.float64)


def store(x, dtype: str):
    """Round to the storage dtype ("bf16" or "f32")."""
    if dtype == "bf16":
        return round_to_bf16(x)
    if dtype == "f32":
        return round_to_f32(x)
    if dtype == "f64":
        return np.asarray(x, dtype=np.float64)
    raise ValueError(dtype)


# --------------------------------------------------------------------------------------
# Slots and blocks  (Sec. 3.2.1 and Sec. 3.3.1)
# --------------------------------------------------------------------------------------


def n_slots(n: int, k: int) -> int:
    """m = ceil(n / k)  (Sec. 3.2.1)."""
    if n < 0 or k < 1:
        raise ValueError("need n >= 0 and k >= 1")
    return -(-n // k)


def block(j: int, n: int, k: int):
    """0-based token range [start, end) of block j.  Sec. 3.3.1 writes the 1-based block
    B(j) = {(j-1)k+1, ..., min(jk, n)}; shifted to 0-based this is [jk, min((j+1)k, n))."""
    return j * k, min((j + 1) * k, n)


def slot_local_positions(n: int, k: int) -> np.ndarray:
    """Position of each slot inside its chunk: the index of the last token of its block
    (Sec. 3.3.1: a C2 token takes the position index of the last token in its block)."""
    return np.array([block(j, n, k)[1] - 1 for j in range(n_slots(n, k))], dtype=np.int64)


# --------------------------------------------------------------------------------------
# RoPE
# --------------------------------------------------------------------------------------


def rope_inv_freq(d: int, theta: float) -> np.ndarray:
    """theta^(-2i/d) for i = 0 .. d/2-1."""
    i = np.arange(d // 2, dtype=np.float64)
    return np.power(float(theta), -2.0 * i / d)


def rope(x, pos, theta: float):
    """Apply RoPE to x[..., T, H, d] at integer positions pos[T] (rotate-half pairing).

    Pair (x_i, x_{i+d/2}) turns by angle pos * theta^(-2i/d):
        x_i'       = x_i cos - x_{i+d/2} sin
        x_{i+d/2}' = x_i sin + x_{i+d/2} cos
    """
    x = np.asarray(x, dtype=np.float64)
    d = x.shape[-1]
    pos = np.asarray(pos, dtype=np.float64)
    ang = pos[:, None] * rope_inv_freq(d, theta)[None, :]          # [T, d/2]
    c = np.cos(ang)[:, None, :]                                      # [T, 1, d/2]
    s = np.sin(ang)[:, None, :]
    x1, x2 = x[..., : d // 2], x[..., d // 2:]
    return np.concatenate([x1 * c - x2 * s, x1 * s + x2 * c], axis=-1)


# --------------------------------------------------------------------------------------
# Compression: the offline encoding step M (Sec. 2.2, Sec. 3.2)
# --------------------------------------------------------------------------------------


def meanpool_slots(tok, k: int):
    """Block means of per-token rows: tok[..., n, H, d] -> [..., m, H, d].

    Adapted from the residual mean-pooling variant (Sec. 3.2.3), which adds the mean of the
    block's hidden states to the C2 token.  The equation there writes 1/k; the last block
    of a chunk whose length is not a multiple of k holds fewer tokens, and this oracle
    divides by the block's true size (a plain mean).
    """
    tok = np.asarray(tok, dtype=np.float64)
    n = tok.shape[-3]
    out = []
    for j in range(n_slots(n, k)):
        a, b = block(j, n, k)
        out.append(tok[..., a:b, :, :].sum(axis=-3) / (b - a))
    return np.stack(out, axis=-3)


def compress_chunk(k_in, v_in, n: int, k: int, theta: float, dtype: str, mode: str):
    """Encode one chunk into its stored slots.

    k_in, v_in: [L, n, H, d] pre-RoPE token K/V for mode "meanpool"; [L, m, H, d] pre-RoPE
    slot K/V for mode "provided" (an external extractor's output).
    Returns (K_stored, V_stored) [L, m, H, d]: K carries RoPE at each slot's local
    position, both rounded to the storage dtype.
    """
    m = n_slots(n, k)
    if mode == "meanpool":
        kb, vb = meanpool_slots(k_in, k), meanpool_slots(v_in, k)
    elif mode == "provided":
        kb, vb = np.asarray(k_in, np.float64), np.asarray(v_in, np.float64)
    else:
        raise ValueError(mode)
    if kb.shape[-3] != m:
        raise ValueError("slot count does not match ceil(n/k)")
    p = slot_local_positions(n, k)
    k_st = np.stack([rope(kb[layer], p, theta) for layer in range(kb.shape[0])])
    return store(k_st, dtype), store(vb, dtype)


# --------------------------------------------------------------------------------------
# Composition: the blending step B (Sec. 2.2; Sec. 3.2.4; Appendix C)
# --------------------------------------------------------------------------------------


def check_positions(lengths, positions):
    """Offsets must be >= 0, non-decreasing, and leave each chunk its full original span."""
    prev_end = 0
    for n, o in zip(lengths, positions):
        if o < 0 or o < prev_end:
            raise ValueError("positions overlap or decrease")
        prev_end = o + n
    return prev_end


def compose(chunks, chunk_ids, positions, theta: float, dtype: str, fixed_pos=False):
    """Compose one request's prefix cache.

    chunks: mapping chunk id -> (K_stored [L, m, H, d], V_stored, n, k)
    chunk_ids, positions: the chunk of each occurrence and its start offset o_i.
    Slot j of occurrence i lands at row D_i + j (D_i = slots of earlier occurrences) with
    composed position o_i + p_j; its K is turned by o_i (from p_j to o_i + p_j), V copied.
    With fixed_pos (the paper's "Fixed-Pos." ablation, Sec. 4.8) nothing is turned and
    slots keep their local positions.
    Returns K [L, S, H, d], V [L, S, H, d], pos [S] (int64), L_req (= max_i o_i + n_i).
    """
    lengths = [chunks[c][2] for c in chunk_ids]
    l_req = check_positions(lengths, positions)
    ks, vs, ps = [], [], []
    for c, o in zip(chunk_ids, positions):
        k_st, v_st, n, k = chunks[c]
        p = slot_local_positions(n, k)
        delta = 0 if fixed_pos else o
        turn = np.full(p.shape, delta, dtype=np.int64)
        ks.append(store(np.stack([rope(k_st[layer], turn, theta)
                                  for layer in range(k_st.shape[0])]), dtype))
        vs.append(np.asarray(v_st, np.float64))
        ps.append(p + delta)
    return (np.concatenate(ks, axis=1), np.concatenate(vs, axis=1),
            np.concatenate(ps), l_req)


def compose_pre_rope(slots, chunk_ids, positions, theta: float):
    """Composition from slots kept before any positional embedding (the storage convention
    Sec. 3.3.1 states): RoPE at o_i + p_j applied once.  No rounding; used to check that
    turning locally-rotated slots by o_i gives the same cache in exact arithmetic.
    slots: mapping chunk id -> (K_pre [L, m, H, d], V [L, m, H, d], n, k)."""
    ks, vs, ps = [], [], []
    for c, o in zip(chunk_ids, positions):
        kb, vb, n, k = slots[c]
        pos = slot_local_positions(n, k) + o
        ks.append(np.stack([rope(kb[layer], pos, theta) for layer in range(kb.shape[0])]))
        vs.append(np.asarray(vb, np.float64))
        ps.append(pos)
    return np.concatenate(ks, axis=1), np.concatenate(vs, axis=1), np.concatenate(ps)


# --------------------------------------------------------------------------------------
# Inference over [KV_total; suffix]  (Sec. 2.2; Sec. 3.2.2 "standard attention operator")
# --------------------------------------------------------------------------------------


def suffix_positions(l_req: int, n_suffix: int) -> np.ndarray:
    """Suffix token t sits at L_req + t, right after the composed span."""
    return l_req + np.arange(n_suffix, dtype=np.int64)


def attend(k_c, v_c, l_req: int, q, k_suf, v_suf, theta: float, dtype: str):
    """Suffix attention for one request.

    k_c, v_c: composed cache [L, S, Hkv, d]; q: [L, Sq, Hq, d]; k_suf, v_suf: [L, Sq, Hkv, d]
    (all pre-RoPE for the suffix).  Suffix Q and K are turned to L_req + t and stored
    (rounded) like any cached activation.  Key j of the sequence [composed; suffix] is
    visible to suffix token t iff j <= S + t.  Scale 1/sqrt(d); exact softmax.
    Returns O [L, Sq, Hq, d] (float64) and lse [L, Hq, Sq] (natural log).
    """
    k_c = np.asarray(k_c, np.float64)
    v_c = np.asarray(v_c, np.float64)
    n_layers, s_len, hkv, d = k_c.shape
    sq, hq = q.shape[1], q.shape[2]
    grp = hq // hkv
    pos = suffix_positions(l_req, sq)
    out = np.zeros((n_layers, sq, hq, d))
    lse = np.zeros((n_layers, hq, sq))
    key_idx = np.arange(s_len + sq)
    visible = key_idx[None, :] <= (s_len + np.arange(sq))[:, None]      # [Sq, S+Sq]
    for layer in range(n_layers):
        q_r = store(rope(q[layer], pos, theta), dtype)
        k_r = store(rope(k_suf[layer], pos, theta), dtype)
        keys = np.concatenate([k_c[layer], k_r], axis=0)               # [S+Sq, Hkv, d]
        vals = np.concatenate([v_c[layer], np.asarray(v_suf[layer], np.float64)], axis=0)
        for h in range(hq):
            g = h // grp
            s = q_r[:, h, :] @ keys[:, g, :].T / math.sqrt(d)          # [Sq, S+Sq]
            s = np.where(visible, s, -np.inf)
            mx = s.max(axis=1, keepdims=True)
            e = np.exp(s - mx)
            tot = e.sum(axis=1, keepdims=True)
            out[layer, :, h, :] = (e / tot) @ vals[:, g, :]
            lse[layer, h, :] = (mx + np.log(tot))[:, 0]
    return out, lse


def decode_step(k_c, v_c, l_req: int, k_prev, v_prev, q_new, k_new, v_new, step: int,
                theta: float, dtype: str):
    """One generation step after the suffix, for one request.

    The new token is suffix token ``step``; suffix tokens 0 .. step-1 (pre-RoPE k_prev,
    v_prev [L, step, Hkv, d]) are already in the cache at positions L_req + t.  The new
    token's q_new [L, Hq, d] and k_new, v_new [L, Hkv, d] (pre-RoPE) sit at L_req + step.
    Its single query row attends to every key: the composed slots k_c, v_c [L, S, Hkv, d]
    and suffix rows 0 .. step (the same standard attention as ``attend``, Sec. 3.2.2, for
    one query; nothing is masked because every cached key precedes it).
    Returns O [L, Hq, d] (float64) and lse [L, Hq] (natural log).
    """
    k_c = np.asarray(k_c, np.float64)
    v_c = np.asarray(v_c, np.float64)
    n_layers, _, hkv, d = k_c.shape
    hq = q_new.shape[1]
    grp = hq // hkv
    prev_pos = suffix_positions(l_req, step)
    out = np.zeros((n_layers, hq, d))
    lse = np.zeros((n_layers, hq))
    for layer in range(n_layers):
        q_r = store(rope(q_new[layer][None], [l_req + step], theta), dtype)[0]      # [Hq, d]
        k_old = store(rope(k_prev[layer], prev_pos, theta), dtype) if step else \
            np.zeros((0, hkv, d))
        k_now = store(rope(k_new[layer][None], [l_req + step], theta), dtype)
        keys = np.concatenate([k_c[layer], k_old, k_now], axis=0)                 # [S+step+1, Hkv, d]
        vals = np.concatenate([v_c[layer], np.asarray(v_prev[layer], np.float64).reshape(-1, hkv, d),
                               np.asarray(v_new[layer], np.float64)[None]], axis=0)
        for h in range(hq):
            g = h // grp
            s = keys[:, g, :] @ q_r[h] / math.sqrt(d)                              # [keys]
            mx = s.max()
            e = np.exp(s - mx)
            tot = e.sum()
            out[layer, h] = (e / tot) @ vals[:, g, :]
            lse[layer, h] = mx + math.log(tot)
    return out, lse


def sif_positions(n: int, k: int) -> np.ndarray:
    """Extraction positions of [x_0 .. x_{n-1}; c_0 .. c_{m-1}] (Sec. 3.3.1): document token
    t at t, C2 token c_j at the last token of its block B(j) = [jk, min((j+1)k, n))."""
    return np.concatenate([np.arange(n), slot_local_positions(n, k)]).astype(np.int64)


def sif_mask(n: int, k: int) -> np.ndarray:
    """Visibility of key u to query t under Structured Information Flow (Sec. 3.3.2), as a
    boolean [n+m, n+m] matrix over [x_0 .. x_{n-1}; c_0 .. c_{m-1}]:
      * original-token invariance: a document token sees document tokens 0..t, never a C2
        token;
      * block-local extraction: c_j sees the document tokens of B(j) and of the sink block;
      * causal accumulation: c_j sees c_0 .. c_j.
    The sink block (B(0) in the paper's 1-based numbering, left undefined by its block
    formula) is read as the first block [0, min(k, n))."""
    m = n_slots(n, k)
    vis = np.zeros((n + m, n + m), dtype=bool)
    for t in range(n):
        vis[t, :t + 1] = True
    for j in range(m):
        lo, hi = block(j, n, k)
        vis[n + j, lo:hi] = True
        s_lo, s_hi = block(0, n, k)
        vis[n + j, s_lo:s_hi] = True
        vis[n + j, n:n + j + 1] = True
    return vis


def sif_attention(q, k_in, v, n: int, k: int, theta: float, dtype: str):
    """One attention layer of the extractor over a chunk under the SIF mask.

    q: [L, n+m, Hq, d], k_in, v: [L, n+m, Hkv, d] (pre-RoPE), ordered
    [document tokens; C2 tokens].  Q and K are turned to ``sif_positions`` and stored
    (rounded) like any cached activation; scale 1/sqrt(d); exact softmax under ``sif_mask``.
    Returns O [L, n+m, Hq, d] (float64) and lse [L, Hq, n+m] (natural log)."""
    n_layers, n_all, hq, d = q.shape
    hkv = k_in.shape[2]
    grp = hq // hkv
    pos = sif_positions(n, k)
    assert len(pos) == n_all
    vis = sif_mask(n, k)
    out = np.zeros((n_layers, n_all, hq, d))
    lse = np.zeros((n_layers, hq, n_all))
    for layer in range(n_layers):
        q_r = store(rope(q[layer], pos, theta), dtype)
        k_r = store(rope(k_in[layer], pos, theta), dtype)
        vals = np.asarray(v[layer], np.float64)
        for h in range(hq):
            g = h // grp
            s = q_r[:, h, :] @ k_r[:, g, :].T / math.sqrt(d)            # [n+m, n+m]
            s = np.where(vis, s, -np.inf)
            mx = s.max(axis=1, keepdims=True)
            e = np.exp(s - mx)
            tot = e.sum(axis=1, keepdims=True)
            out[layer, :, h, :] = (e / tot) @ vals[:, g, :]
            lse[layer, h, :] = (mx + np.log(tot))[:, 0]
    return out, lse


def attend_partial(keys, vals, q_r, visible):
    """Attention of rotated queries q_r [Sq, Hq, d] over an explicit key set
    keys/vals [T, Hkv, d] with a boolean visibility mask [Sq, T]; returns (O, lse) with
    lse = -inf where a row sees no key (its O is then 0)."""
    sq, hq, d = q_r.shape
    grp = hq // keys.shape[1]
    out = np.zeros((sq, hq, d))
    lse = np.full((hq, sq), -np.inf)
    for h in range(hq):
        g = h // grp
        s = np.where(visible, q_r[:, h, :] @ keys[:, g, :].T / math.sqrt(d), -np.inf)
        for t in range(sq):
            if not visible[t].any():
                continue
            mx = s[t].max()
            e = np.exp(s[t] - mx)
            out[t, h] = e @ vals[:, g, :] / e.sum()
            lse[h, t] = mx + math.log(e.sum())
    return out, lse


def lse_combine(outs, lses):
    """Merge attention over disjoint key sets: lse = log sum_s exp(lse_s),
    O = sum_s exp(lse_s - lse) O_s.  outs: list of [Sq, Hq, d]; lses: list of [Hq, Sq]."""
    lses = np.stack(lses)                               # [P, Hq, Sq]
    mx = np.max(lses, axis=0)
    w = np.exp(lses - mx[None])
    tot = w.sum(axis=0)
    lse = mx + np.log(tot)
    wt = (w / tot[None]).transpose(0, 2, 1)[..., None]  # [P, Sq, Hq, 1]
    return (np.stack(outs) * wt).sum(axis=0), lse


# --------------------------------------------------------------------------------------
# A whole batch, as the library sees it
# --------------------------------------------------------------------------------------


def run_request(chunks, chunk_ids, positions, q, k_suf, v_suf, theta, dtype, fixed_pos=False):
    """compose + attend for one request; returns a dict of every intermediate."""
    k_c, v_c, pos, l_req = compose(chunks, chunk_ids, positions, theta, dtype, fixed_pos)
    o, lse = attend(k_c, v_c, l_req, q, k_suf, v_suf, theta, dtype)
    return dict(k=k_c, v=v_c, pos=pos, l_req=l_req, out=o, lse=lse)
