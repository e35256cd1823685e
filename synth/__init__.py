"""Seeded synthetic inputs for the C2KV compose + suffix-attention path.

This module only draws random numbers and lays out request structure (which chunks a
request reuses and at which offsets).  It holds none of the method's arithmetic: no
pooling, no RoPE, no composition, no attention.  Both the CPU oracle and the CUDA path
are fed from here, so neither ever sees an input the other produced.

Inputs stand in for the paper's LongBench / RULER documents (Sec. 4.1), which are not
available: K/V rows are N(0, 1) with a few outlier channels scaled up, the way real
key caches show a handful of large-magnitude channels.

Workload shapes
---------------
``tiny_f32``      1 layer, Hq 4 / Hkv 2, d 64, theta 1e4, fp32; 4 chunks x 128 tokens,
                  ratio 4, offsets 0/128/256/384, 32 suffix tokens.
``llama8b``       Llama-3-8B layer: Hq 32 / Hkv 8, d 128, theta 5e5, bf16; 10 chunks x 512
                  tokens, ratio 4 (5120 composed positions), 64 suffix tokens, batch 1;
                  32 layers when timed as a whole model (``llama8b_l1``: one layer).
``batched``       pool of 256 chunks x 512 tokens (ratio 4); 16 requests, each 8 distinct
                  chunks drawn Zipf(s=1.1), random order; 128 suffix tokens.
``long70b``       Llama-3-70B layer: Hq 64 / Hkv 8, d 128; 32 chunks x 1024 tokens,
                  ratio 16 (32768 positions), 256 suffix tokens, batch 2.
``sweep_k{k}``    Llama-3-8B layer; 8 requests x 16 chunks x 2048 tokens, 128 suffix
                  tokens; k in {1 (uncompressed control), 4, 8, 10, 16}.
"""
from __future__ import annotations

import dataclasses

import numpy as np

__all__ = [
    "Workload", "WORKLOADS", "workload", "round_f32_to_bf16", "chunk_tokens",
    "chunk_slots", "requests", "suffix", "scaled", "outlier_mask",
]

SWEEP_RATIOS = (1, 4, 8, 10, 16)


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    layers: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    rope_theta: float
    dtype: str                # "bf16" or "f32"
    chunk_tokens: int         # tokens per precomputed chunk (n)
    ratio_k: int              # compression ratio k (slots = ceil(n/k))
    n_suffix: int             # suffix / query tokens per request
    batch: int                # concurrent requests
    chunks_per_request: int
    pool_chunks: int          # distinct chunks precomputed
    draw: str                 # "in_order" | "zipf" | "distinct"
    zipf_s: float = 1.1
    outlier: str = "frac"     # "fixed4": 4 channels shared by all heads; "frac": 2% of (head, ch)
    outlier_scale: float = 10.0
    outlier_frac: float = 0.02
    gap: int = 0              # tokens left free before each chunk (static/system context)

    @property
    def group(self) -> int:
        return self.n_q_heads // self.n_kv_heads


WORKLOADS = {
    "tiny_f32": Workload("tiny_f32", 1, 4, 2, 64, 1.0e4, "f32", 128, 4, 32, 1, 4, 4,
                         "in_order", outlier="fixed4", outlier_scale=8.0),
    "llama8b": Workload("llama8b", 32, 32, 8, 128, 5.0e5, "bf16", 512, 4, 64, 1, 10, 10,
                        "in_order"),
    "batched": Workload("batched", 1, 32, 8, 128, 5.0e5, "bf16", 512, 4, 128, 16, 8, 256,
                        "zipf"),
    "long70b": Workload("long70b", 1, 64, 8, 128, 5.0e5, "bf16", 1024, 16, 256, 2, 32, 64,
                        "distinct"),
}
# the same Llama-3-8B workload timed one layer at a time (per-layer TTFT proxy)
WORKLOADS["llama8b_l1"] = dataclasses.replace(WORKLOADS["llama8b"], name="llama8b_l1", layers=1)
for _k in SWEEP_RATIOS:
    WORKLOADS[f"sweep_k{_k}"] = Workload(f"sweep_k{_k}", 1, 32, 8, 128, 5.0e5, "bf16", 2048,
                                         _k, 128, 8, 16, 128, "distinct")


def workload(name: str) -> Workload:
    return WORKLOADS[name]


def scaled(wl: Workload, **changes) -> Workload:
    """A copy of ``wl`` with some fields replaced (for reduced parity cases)."""
    return dataclasses.replace(wl, **changes)


def round_f32_to_bf16(x: np.ndarray) -> np.ndarray:
    """Round float32 values to the nearest bfloat16 (ties to even); returns float32.

    Used only to make generated inputs exactly representable in the storage type, so that
    every consumer sees identical input bits.
    """
    x = np.ascontiguousarray(x, dtype=np.float32)
    bits = x.view(np.uint32).astype(np.uint64)
    bias = ((bits >> 16) & 1) + 0x7FFF
    out = ((bits + bias) & 0xFFFF0000).astype(np.uint32)
    return out.view(np.float32)


def _rng(seed: int, *stream: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([seed, *stream])))


_TAG_OUTLIER, _TAG_CHUNK, _TAG_SLOTS, _TAG_REQ, _TAG_SUFFIX, _TAG_EXTRACT = 1, 2, 3, 4, 5, 6


def outlier_mask(wl: Workload, seed: int = 0) -> np.ndarray:
    """Per-(head, channel) multiplier [Hkv, d]: 1 everywhere except the outlier channels."""
    rng = _rng(seed, _TAG_OUTLIER)
    mult = np.ones((wl.n_kv_heads, wl.head_dim), dtype=np.float32)
    if wl.outlier == "fixed4":
        ch = rng.choice(wl.head_dim, size=4, replace=False)
        mult[:, ch] = wl.outlier_scale
    else:
        count = int(round(wl.outlier_frac * wl.n_kv_heads * wl.head_dim))
        flat = rng.choice(wl.n_kv_heads * wl.head_dim, size=count, replace=False)
        mult.reshape(-1)[flat] = wl.outlier_scale
    return mult


def _finish(x: np.ndarray, dtype: str) -> np.ndarray:
    return round_f32_to_bf16(x) if dtype == "bf16" else np.ascontiguousarray(x, np.float32)


def chunk_tokens(wl: Workload, chunk_id: int, seed: int = 0, n_tokens: int | None = None):
    """Pre-RoPE per-token K and V of one chunk, shape [layers, n, Hkv, d] (float32 holding
    values exact in the workload dtype)."""
    n = wl.chunk_tokens if n_tokens is None else n_tokens
    rng = _rng(seed, _TAG_CHUNK, chunk_id)
    shape = (wl.layers, n, wl.n_kv_heads, wl.head_dim)
    mult = outlier_mask(wl, seed)
    k = rng.standard_normal(shape, dtype=np.float32) * mult
    v = rng.standard_normal(shape, dtype=np.float32) * mult
    return _finish(k, wl.dtype), _finish(v, wl.dtype)


def chunk_slots(wl: Workload, chunk_id: int, n_slots: int, seed: int = 0):
    """Random stand-ins for already-stored compressed slots, [layers, m, Hkv, d]: what a
    storage tier would hand back for a chunk (used by the load / STORED path)."""
    rng = _rng(seed, _TAG_SLOTS, chunk_id)
    shape = (wl.layers, n_slots, wl.n_kv_heads, wl.head_dim)
    mult = outlier_mask(wl, seed)
    k = rng.standard_normal(shape, dtype=np.float32) * mult
    v = rng.standard_normal(shape, dtype=np.float32) * mult
    return _finish(k, wl.dtype), _finish(v, wl.dtype)


def requests(wl: Workload, seed: int = 0):
    """Request structure: for each request, the list of pool chunk ids it reuses (in
    composition order) and their start offsets in the composed sequence.

    Offsets accumulate over the uncompressed chunk lengths, plus ``wl.gap`` free positions
    before each chunk (room for a static / system prompt).
    """
    rng = _rng(seed, _TAG_REQ)
    out = []
    for r in range(wl.batch):
        if wl.draw == "in_order":
            ids = list(range(wl.chunks_per_request))
        elif wl.draw == "distinct":
            ids = list(range(r * wl.chunks_per_request, (r + 1) * wl.chunks_per_request))
            ids = [i % wl.pool_chunks for i in ids]
        elif wl.draw == "zipf":
            ranks = np.arange(1, wl.pool_chunks + 1, dtype=np.float64)
            p = ranks ** (-wl.zipf_s)
            p /= p.sum()
            ids = rng.choice(wl.pool_chunks, size=wl.chunks_per_request, replace=False, p=p)
            ids = [int(i) for i in rng.permutation(ids)]
        else:
            raise ValueError(wl.draw)
        offsets, o = [], 0
        for _ in ids:
            o += wl.gap
            offsets.append(o)
            o += wl.chunk_tokens
        out.append((ids, offsets))
    return out


def suffix(wl: Workload, seed: int = 0, layers: int | None = None):
    """Pre-RoPE suffix tensors: q [layers, B, Sq, Hq, d], k/v [layers, B, Sq, Hkv, d]."""
    L = wl.layers if layers is None else layers
    rng = _rng(seed, _TAG_SUFFIX)
    q = rng.standard_normal((L, wl.batch, wl.n_suffix, wl.n_q_heads, wl.head_dim),
                            dtype=np.float32)
    k = rng.standard_normal((L, wl.batch, wl.n_suffix, wl.n_kv_heads, wl.head_dim),
                            dtype=np.float32)
    v = rng.standard_normal((L, wl.batch, wl.n_suffix, wl.n_kv_heads, wl.head_dim),
                            dtype=np.float32)
    return _finish(q, wl.dtype), _finish(k, wl.dtype), _finish(v, wl.dtype)




def extraction_inputs(wl: Workload, chunk_id: int, n_tokens: int, ratio_k: int, seed: int = 0):
    """Inputs of one extraction attention layer over a chunk: q [layers, n+m, Hq, d] and
    k, v [layers, n+m, Hkv, d] (pre-RoPE), ordered [document tokens; m = ceil(n/k) C2
    tokens].  The document K/V are the chunk's own tokens (``chunk_tokens``); the queries
    and the C2 tokens' K/V, which trained projections would make, are standard normal."""
    n = n_tokens
    m = -(-n // ratio_k)
    kd, vd = chunk_tokens(wl, chunk_id, seed, n_tokens=n)
    rng = _rng(seed, _TAG_EXTRACT, chunk_id)
    q = rng.standard_normal((wl.layers, n + m, wl.n_q_heads, wl.head_dim), dtype=np.float32)
    kc = rng.standard_normal((wl.layers, m, wl.n_kv_heads, wl.head_dim), dtype=np.float32)
    vc = rng.standard_normal((wl.layers, m, wl.n_kv_heads, wl.head_dim), dtype=np.float32)
    k = np.concatenate([kd, _finish(kc, wl.dtype)], axis=1)
    v = np.concatenate([vd, _finish(vc, wl.dtype)], axis=1)
    return _finish(q, wl.dtype), k, v
