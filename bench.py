"""Benchmark of the C2KV hot path: compose stored compressed chunks into one GQA cache
(RoPE re-rotated) and run the suffix tokens' attention over it, through the C ABI.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                    [--workload NAME]

A step is one pass of the whole path over one batch: c2kv_compose (all layers, one
launch) + c2kv_attend (suffix RoPE/append + attention, all layers) + cache release.
Metric: composed KV tokens/s = composed positions of the batch / step time.
Prints one JSON line (rank 0).  Under torchrun every rank runs its own replica of the
workload (requests are independent: weak scaling, no data-path collective); only the
timing barrier and the max-over-ranks reduction cross ranks.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import synth  # noqa: E402

L2_FLUSH_BYTES = 256 << 20          # > 129 MB of L2
METRIC = "composed KV tokens/s"


# --------------------------------------------------------------------------- workload

def workload_facts(wl):
    """Sizes the metric and the rooflines are computed from."""
    m = -(-wl.chunk_tokens // wl.ratio_k)
    S = wl.chunks_per_request * m                          # composed slots / request
    span = wl.chunks_per_request * (wl.chunk_tokens + wl.gap)
    eb = 4 if wl.dtype == "f32" else 2
    row_bytes = wl.n_kv_heads * wl.head_dim * eb
    # compose: every stored slot read once (K and V) and written once, plus its position
    compose_bytes = wl.layers * wl.batch * S * row_bytes * 2 * 2 + wl.batch * S * 4
    sq = wl.n_suffix
    keys = S * sq + sq * (sq + 1) // 2                     # visible (query, key) pairs
    attn_flops = 4 * wl.head_dim * wl.n_q_heads * keys * wl.batch * wl.layers
    # attention bytes: every cache row (slots + suffix) read once, Q read, O written
    attn_bytes = wl.layers * wl.batch * ((S + sq) * row_bytes * 2
                                         + 2 * sq * wl.n_q_heads * wl.head_dim * eb)
    # fused compose + suffix preparation + attention (one kernel): every stored slot read and
    # its composed row written once (compose's bytes), the suffix rows read and written to the
    # cache once, Q read, O written; the cache is not read back
    fused_bytes = compose_bytes + wl.layers * wl.batch * (2 * sq * row_bytes * 2
                                                          + 2 * sq * wl.n_q_heads * wl.head_dim * eb)
    return dict(name=wl.name, slots=S, span=span, positions=wl.batch * span, row_bytes=row_bytes, dtype=wl.dtype,
                compose_bytes=compose_bytes, attn_flops=attn_flops, attn_bytes=attn_bytes,
                fused_bytes=fused_bytes,
                slots_per_chunk=m)


def describe(wl):
    f = workload_facts(wl)
    return (f"{wl.name}: Hq{wl.n_q_heads}/Hkv{wl.n_kv_heads} d{wl.head_dim} {wl.dtype}, "
            f"{wl.layers} layers, batch {wl.batch} x {wl.chunks_per_request} chunks x "
            f"{wl.chunk_tokens} tok, k={wl.ratio_k} ({f['slots']} slots, {f['span']} "
            f"positions/request), {wl.n_suffix} suffix tokens")


def source_digest(paths):
    """First 16 hex digits of the sha256 of the given C++/CUDA source files, concatenated in
    order, with comments and blank lines removed (so that a comment edit does not count as a
    change of the kernel)."""
    import hashlib
    import re
    h = hashlib.sha256()
    for rel in paths:
        with open(os.path.join(ROOT, rel), encoding="utf-8") as fh:
            text = fh.read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        text = re.sub(r"//[^\n]*", "", text)
        code = "\n".join(line.rstrip() for line in text.splitlines() if line.strip())
        h.update(code.encode("utf-8"))
    return h.hexdigest()[:16]


def captured_traffic(kernel, workload):
    """DRAM bytes per launch from the committed ncu summary, if it was captured on this
    workload and every source the kernel is built from is still the one that was captured
    (else None: the counters do not describe this launch).  Records are keyed
    "kernel@workload" (or "kernel" for the default workload's)."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(path):
        return None
    with open(path) as fh:
        recs = json.load(fh)
    rec = recs.get(f"{kernel}@{workload}") or recs.get(kernel)
    if not rec or "sources" not in rec or rec.get("workload") != workload:
        return None
    return rec["traffic_bytes"] if source_digest(rec["sources"]) == rec["sha256_16"] else None


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as fh:
            pk = json.load(fh)
        return pk["hbm_gbs"], pk["bf16_tflops"], pk.get("bf16_tflops_sustained"), "measured"
    return 6800.0, 1900.0, 1700.0, "fallback"


def rooflines(compose_ms, attn_ms, f, hbm, bf16, src):
    """Roofline objects for the compose kernel and the attention kernel (algorithmic work /
    measured kernel time), with the dominant one as "roofline"."""
    comp_gbs = f["compose_bytes"] / (compose_ms / 1e3) / 1e9
    compose = {"bound": "hbm", "kernel": "compose_bulk_kernel", "achieved": round(comp_gbs, 1),
               "peak": hbm, "unit": "GB/s", "frac": round(comp_gbs / hbm, 4),
               "traffic": captured_traffic("compose_kernel", f["name"]), "peak_source": f"{src} hbm_gbs",
               "bytes_per_launch": f["compose_bytes"]}
    intensity = f["attn_flops"] / f["attn_bytes"]
    ridge = bf16 * 1e12 / (hbm * 1e9)
    attn_tfs = f["attn_flops"] / (attn_ms / 1e3) / 1e12
    attn_gbs = f["attn_bytes"] / (attn_ms / 1e3) / 1e9
    if intensity < ridge:
        attend = {"bound": "hbm", "achieved": round(attn_gbs, 1), "peak": hbm, "unit": "GB/s",
                  "frac": round(attn_gbs / hbm, 4), "peak_source": f"{src} hbm_gbs",
                  "bytes_per_launch": f["attn_bytes"]}
    else:
        attend = {"bound": "tensor", "achieved": round(attn_tfs, 2), "peak": bf16,
                  "unit": "TFLOP/s", "frac": round(attn_tfs / bf16, 4),
                  "peak_source": f"{src} bf16_tflops (burst)", "flops_per_launch": f["attn_flops"]}
    if f.get("dtype") == "f32":
        # fp32 attention runs on the CUDA cores (attn_simt_kernel): plain FP32 FMA arithmetic,
        # against 128 FMA lanes x 2 flop x 152 SMs x 2.07 GHz = 80.5 TFLOP/s
        alu = 128 * 2 * 152 * 2.07e9 / 1e12
        return {"roofline": {"bound": "alu", "kernel": "attn_simt_kernel", "achieved": round(attn_tfs, 3),
                             "peak": round(alu, 1), "unit": "TFLOP/s", "frac": round(attn_tfs / alu, 4),
                             "peak_source": "derived: FP32 FMA lanes x clock", "traffic": None,
                             "flops_per_launch": f["attn_flops"]},
                "roofline_compose": compose}
    attend.update({"kernel": "attn_tc_kernel", "traffic": captured_traffic("attn_tc_kernel", f["name"]),
                   "intensity_flop_per_byte": round(intensity, 1), "ridge": round(ridge, 1),
                   "tensor_frac": round(attn_tfs / bf16, 4), "hbm_frac": round(attn_gbs / hbm, 4)})
    if attn_ms >= compose_ms:
        return {"roofline": attend, "roofline_compose": compose}
    return {"roofline": compose, "roofline_attend": attend}


def step_rooflines(fused_ran, kern, kc_ms, ka_ms, f, hbm, bf16, src):
    r = rooflines(kc_ms, ka_ms, f, hbm, bf16, src)
    if not fused_ran:
        return r
    parts = {o["kernel"]: o for o in r.values()}
    return {"roofline": fused_roofline(kern["fused"][0], f, hbm, bf16, src),
            "roofline_compose": parts.get("compose_bulk_kernel"),
            "roofline_attend": parts.get("attn_tc_kernel", parts.get("attn_simt_kernel"))}


def fused_roofline(fused_ms, f, hbm, bf16, src):
    """The fused compose + suffix preparation + attention kernel: HBM-bound (its intensity,
    attention flops over fused bytes, is far below the ridge); both fractions carried."""
    gbs = f["fused_bytes"] / (fused_ms / 1e3) / 1e9
    tfs = f["attn_flops"] / (fused_ms / 1e3) / 1e12
    return {"bound": "hbm", "kernel": "attn_tc_kernel<fused>",
            "achieved": round(gbs, 1), "peak": hbm, "unit": "GB/s", "frac": round(gbs / hbm, 4),
            "peak_source": f"{src} hbm_gbs", "bytes_per_launch": f["fused_bytes"],
            "traffic": captured_traffic("attn_tc_kernel_fused", f["name"]),
            "intensity_flop_per_byte": round(f["attn_flops"] / f["fused_bytes"], 1),
            "tensor_frac": round(tfs / bf16, 4), "hbm_frac": round(gbs / hbm, 4)}


# --------------------------------------------------------------------------- clocks

class ClockSampler:
    """nvidia-smi sampling of SM clocks and throttle reasons while the timed region runs."""

    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.proc = None
        self.gpu = gpu_index
        self.path = os.path.join("/tmp", f"c2kv_clocks_{os.getpid()}.csv")

    def __enter__(self):
        try:
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.QUERY}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=self.fh, stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except (OSError, FileNotFoundError):
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.fh.close()

    def summary(self):
        if self.proc is None or not os.path.exists(self.path):
            return None
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
            except ValueError:
                continue
            for name, val in zip(names, parts[5:9]):
                if val.lower().startswith("active"):
                    reasons.add(name)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(smax),
                "reasons": sorted(reasons), "samples": len(sm)}


# --------------------------------------------------------------------------- our arm

class Arm:
    """This rank's share of the global batch (wl.batch requests per rank) on its GPU."""

    def __init__(self, wl, rank, world, torch, c2kv, attn_split=0):
        from paper_2607_17715_gb300.shard import shard_range
        seed = 0
        gwl = synth.scaled(wl, batch=wl.batch * world)
        all_reqs = synth.requests(gwl, seed)
        a, b = shard_range(len(all_reqs), rank, world)
        wl = synth.scaled(wl, batch=b - a)
        self.wl, self.torch, self.c2kv = wl, torch, c2kv
        f = self.facts = workload_facts(wl)
        self.tdt = torch.float32 if wl.dtype == "f32" else torch.bfloat16
        self.stream = torch.cuda.current_stream()
        self.reqs = all_reqs[a:b]
        pool_ids = sorted({c for ids, _ in self.reqs for c in ids})
        m = f["slots_per_chunk"]
        self.ctx = c2kv.c2kv_create(
            wl.layers, wl.n_q_heads, wl.n_kv_heads, wl.head_dim, wl.rope_theta,
            c2kv.DTYPE_F32 if wl.dtype == "f32" else c2kv.DTYPE_BF16,
            pool_slots=len(pool_ids) * m * 2 + 64, stream=self.stream, attn_split=attn_split)
        # stored compressed chunks, kept in pinned host memory (the storage tier) and
        # loaded once into the device pool for the device-resident measurement
        self.host_chunks = {}
        self.dev_ids = {}
        for cid in pool_ids:
            ks, vs = synth.chunk_slots(wl, cid, m, seed)
            kh = torch.from_numpy(ks).to(self.tdt).pin_memory()
            vh = torch.from_numpy(vs).to(self.tdt).pin_memory()
            self.host_chunks[cid] = (kh, vh)
            self.dev_ids[cid] = c2kv.c2kv_compress_chunk(self.ctx, kh, vh, wl.chunk_tokens,
                                                         wl.ratio_k, c2kv.MODE_STORED)
        # the same pinned slots registered in place (MODE_HOST: no copy, no pool slots);
        # compose then reads them from host memory over the CPU-GPU link every step
        self.host_ids = {cid: c2kv.c2kv_compress_chunk(self.ctx, kh, vh, wl.chunk_tokens,
                                                       wl.ratio_k, c2kv.MODE_HOST)
                         for cid, (kh, vh) in self.host_chunks.items()}
        self.req_ptr = np.cumsum([0] + [len(ids) for ids, _ in self.reqs]).astype(np.int32)
        self.positions = [o for _, offs in self.reqs for o in offs]
        q, k, v = synth.suffix(gwl, seed)
        self.q_host = [torch.from_numpy(np.ascontiguousarray(x[:, a:b])).to(self.tdt).pin_memory()
                       for x in (q, k, v)]
        self.q_dev = [x.to("cuda") for x in self.q_host]
        self.out = torch.empty_like(self.q_dev[0])
        self.out_host = torch.empty(self.out.shape, dtype=self.tdt).pin_memory()
        self.flush_buf = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device="cuda")
        c2kv.c2kv_sync(self.ctx)

    def flush_l2(self):
        self.flush_buf.fill_(1.0)

    def compose_warm(self, steps):
        """Median time of c2kv_compose right after an identical compose (no L2 flush: the
        inputs stay in L2 where they fit), event-timed around the call."""
        c2kv, wl, E = self.c2kv, self.wl, self.torch.cuda.Event
        ids = [self.dev_ids[c] for ids_, _ in self.reqs for c in ids_]
        evs = []
        for _ in range(steps):
            c2kv.c2kv_cache_release(self.ctx, c2kv.c2kv_compose(self.ctx, self.req_ptr, ids,
                                                                self.positions, wl.n_suffix))
            a, b = E(enable_timing=True), E(enable_timing=True)
            a.record(self.stream)
            cache = c2kv.c2kv_compose(self.ctx, self.req_ptr, ids, self.positions, wl.n_suffix)
            b.record(self.stream)
            c2kv.c2kv_cache_release(self.ctx, cache)
            evs.append((a, b))
        self.torch.cuda.synchronize()
        return statistics.median(a.elapsed_time(b) for a, b in evs)

    def step_device(self, ev, fused=True):
        """One step with inputs resident in HBM: c2kv_compose_attend (the library fuses the
        two when that pays), or c2kv_compose then c2kv_attend; then the cache is released.
        ev = 4 events: before the step and after the release; on the unfused route also
        after compose and after attend.  The joint call records nothing in between: an event
        recorded between the call and the release of the cache's memory delays the step's
        end by about 4 us on a GB300 (97.5 against 93.2 us on the 32-layer step)."""
        c2kv, wl = self.c2kv, self.wl
        ids = [self.dev_ids[c] for ids_, _ in self.reqs for c in ids_]
        ev[0].record(self.stream)
        if fused:
            cache = c2kv.c2kv_compose_attend(self.ctx, self.req_ptr, ids, self.positions,
                                             wl.n_suffix, *self.q_dev, wl.n_suffix, self.out)
        else:
            cache = c2kv.c2kv_compose(self.ctx, self.req_ptr, ids, self.positions, wl.n_suffix)
            ev[1].record(self.stream)
            c2kv.c2kv_attend(self.ctx, cache, -1, *self.q_dev, wl.n_suffix, self.out)
            ev[2].record(self.stream)
        c2kv.c2kv_cache_release(self.ctx, cache)
        ev[3].record(self.stream)

    def step_e2e_host(self):
        """The same step from host buffers, zero-copy: one call whose kernels read the chunks'
        pinned host slots (compose: load, re-rotation and gather in one kernel) and the
        suffix Q/K/V from pinned host memory, and write O into pinned host memory, across the
        CPU-GPU link (host-resident chunks take compose, then attention, in layer groups)."""
        c2kv, wl = self.c2kv, self.wl
        ids = [self.host_ids[c] for ids_, _ in self.reqs for c in ids_]
        cache = c2kv.c2kv_compose_attend(self.ctx, self.req_ptr, ids, self.positions, wl.n_suffix,
                                         *self.q_host, wl.n_suffix, self.out_host)
        c2kv.c2kv_cache_release(self.ctx, cache)

    def step_e2e(self):
        """The same step from host buffers, staged: copy the requested chunks from pinned host
        memory into the pool, copy the suffix in, compose and attend (one call), read the
        output back."""
        c2kv, wl, torch = self.c2kv, self.wl, self.torch
        loaded = {}
        for cid, (kh, vh) in self.host_chunks.items():
            loaded[cid] = c2kv.c2kv_compress_chunk(self.ctx, kh, vh, wl.chunk_tokens,
                                                   wl.ratio_k, c2kv.MODE_STORED)
        qd = [x.to("cuda", non_blocking=True) for x in self.q_host]
        ids = [loaded[c] for ids_, _ in self.reqs for c in ids_]
        cache = c2kv.c2kv_compose_attend(self.ctx, self.req_ptr, ids, self.positions, wl.n_suffix,
                                         *qd, wl.n_suffix, self.out)
        self.out_host.copy_(self.out, non_blocking=True)
        c2kv.c2kv_cache_release(self.ctx, cache)
        for cid in loaded.values():
            c2kv.c2kv_free_chunk(self.ctx, cid)

    def decode_run(self, steps, warmup, events):
        ids = [self.dev_ids[c] for ids_, _ in self.reqs for c in ids_]
        return decode_measure(self.c2kv, self.torch, self.ctx, self.wl, self.stream, self.req_ptr, ids,
                              self.positions, self.q_dev, self.out, steps, warmup, events, self.flush_l2)

    def extract_run(self, steps, warmup, events):
        """Extraction attention over one chunk of the workload's size (n tokens, ratio k, all
        layers in one call), L2 flushed before each call (untimed).  The inputs are drawn on
        the device: the timing does not depend on their values.  Returns (mean ms per call,
        mean ms of the library's trace of the call)."""
        c2kv, wl, torch = self.c2kv, self.wl, self.torch
        n, k = wl.chunk_tokens, wl.ratio_k
        n_all = n + -(-n // k)
        gen = torch.Generator(device="cuda").manual_seed(2)
        q = torch.randn((wl.layers, n_all, wl.n_q_heads, wl.head_dim), device="cuda", generator=gen).to(self.tdt)
        kk = torch.randn((wl.layers, n_all, wl.n_kv_heads, wl.head_dim), device="cuda", generator=gen).to(self.tdt)
        v = torch.randn_like(kk)
        out = torch.empty_like(q)
        for _ in range(warmup):
            self.flush_l2()
            c2kv.c2kv_extract_attention(self.ctx, wl.layers, q, kk, v, n, k, out)
        c2kv.c2kv_sync(self.ctx)
        for i in range(steps):
            self.flush_l2()                                    # untimed
            events[i][0].record(self.stream)
            c2kv.c2kv_extract_attention(self.ctx, wl.layers, q, kk, v, n, k, out)
            events[i][1].record(self.stream)
        torch.cuda.synchronize()
        c2kv.c2kv_sync(self.ctx)
        ms = sum(ev[0].elapsed_time(ev[1]) for ev in events[:steps]) / steps
        c2kv.c2kv_profile_read(self.ctx)
        c2kv.c2kv_profile_enable(self.ctx, True)
        for i in range(steps):
            self.flush_l2()
            c2kv.c2kv_extract_attention(self.ctx, wl.layers, q, kk, v, n, k, out)
        kern = c2kv.c2kv_profile_read(self.ctx)
        c2kv.c2kv_profile_enable(self.ctx, False)
        return ms, kern["extract"][0]

    def e2e_bytes(self, zero_copy=False):
        """Host->device and device->host bytes of one e2e step.  Staged: each distinct
        chunk is copied once.  Zero-copy: compose reads a chunk's slots once per occurrence."""
        size = {c: kh.numel() * kh.element_size() * 2 for c, (kh, _) in self.host_chunks.items()}
        if zero_copy:
            h2d = sum(size[c] for ids_, _ in self.reqs for c in ids_)
        else:
            h2d = sum(size.values())
        h2d += sum(x.numel() * x.element_size() for x in self.q_host)
        d2h = self.out_host.numel() * self.out_host.element_size()
        return h2d, d2h

    def close(self):
        self.c2kv.c2kv_destroy(self.ctx)


def decode_measure(c2kv, torch, ctx, wl, stream, req_ptr, ids, positions, q_dev, out, steps, warmup,
                   events, flush):
    """Decode after the suffix: compose once, write the suffix with attend, then decode
    `warmup` untimed and `steps` timed tokens per request (one c2kv_decode call per token,
    all layers), L2 flushed before each; then `steps` more tokens with the library's trace
    on, for the decode kernel's own time.  Returns (ms per timed step, mean decode kernel ms
    from the trace, keys read per timed step summed over requests, list of step ms)."""
    tdt = torch.float32 if wl.dtype == "f32" else torch.bfloat16
    cache = c2kv.c2kv_compose(ctx, req_ptr, ids, positions, wl.n_suffix + warmup + 2 * steps)
    c2kv.c2kv_attend(ctx, cache, -1, *q_dev, wl.n_suffix, out)
    B = len(req_ptr) - 1
    gen = torch.Generator(device="cuda").manual_seed(1)
    qd = torch.randn((wl.layers, B, wl.n_q_heads, wl.head_dim), device="cuda", generator=gen).to(tdt)
    kd = torch.randn((wl.layers, B, wl.n_kv_heads, wl.head_dim), device="cuda", generator=gen).to(tdt)
    vd = torch.randn_like(kd)
    od = torch.empty_like(qd)
    n_slots = c2kv.c2kv_cache_info(cache)["n_slots"]
    for i in range(warmup):
        flush()
        c2kv.c2kv_decode(ctx, cache, -1, qd, kd, vd, [wl.n_suffix + i] * B, od)
    c2kv.c2kv_sync(ctx)
    keys = 0
    for i in range(steps):
        st = wl.n_suffix + warmup + i
        flush()                                            # untimed
        events[i][0].record(stream)
        c2kv.c2kv_decode(ctx, cache, -1, qd, kd, vd, [st] * B, od)
        events[i][1].record(stream)
        keys += int(sum(int(n) + st + 1 for n in n_slots))
    torch.cuda.synchronize()
    c2kv.c2kv_sync(ctx)
    per = [ev[0].elapsed_time(ev[1]) for ev in events[:steps]]
    c2kv.c2kv_profile_read(ctx)
    c2kv.c2kv_profile_enable(ctx, True)
    for i in range(steps):
        flush()
        c2kv.c2kv_decode(ctx, cache, -1, qd, kd, vd, [wl.n_suffix + warmup + steps + i] * B, od)
    kern = c2kv.c2kv_profile_read(ctx)
    c2kv.c2kv_profile_enable(ctx, False)
    c2kv.c2kv_sync(ctx)
    c2kv.c2kv_cache_release(ctx, cache)
    return sum(per) / steps, kern["decode"][0], keys / steps, per


def sif_visible_pairs(n, k):
    """(query, key) pairs the Structured Information Flow mask lets through over
    [n document tokens; m = ceil(n/k) C2 tokens]: document token t sees t + 1 keys; C2
    token c_j sees its block, the first (sink) block when j > 0, and c_0 .. c_j."""
    m = -(-n // k)
    sink = min(k, n)
    pairs = n * (n + 1) // 2
    for j in range(m):
        blk = min((j + 1) * k, n) - j * k
        pairs += blk + (sink if j > 0 else 0) + j + 1
    return pairs


def extract_line(wl, world, ms, kernel_ms, hbm, bf16, src):
    """Extraction attention over one chunk per rank: document tokens/s over the job, and the
    call against the tensor and HBM rooflines (algorithmic flops: 4 d per visible (query
    head, key) pair; bytes: Q, K, V read and O written once)."""
    eb = 4 if wl.dtype == "f32" else 2
    n, k = wl.chunk_tokens, wl.ratio_k
    n_all = n + -(-n // k)
    flops = 4.0 * wl.head_dim * wl.n_q_heads * sif_visible_pairs(n, k) * wl.layers
    nbytes = n_all * (2 * wl.n_q_heads + 2 * wl.n_kv_heads) * wl.head_dim * eb * wl.layers
    t = (kernel_ms or ms) / 1e3
    tfs, gbs = flops / t / 1e12, nbytes / t / 1e9
    ridge = bf16 * 1e12 / (hbm * 1e9)
    tensor = flops / nbytes >= ridge
    return {
        "metric": "extracted document tokens/s", "unit": "tokens/s",
        "value": round(n * world / (ms / 1e3), 1), "ms_per_call": round(ms, 5),
        "what": f"c2kv_extract_attention over one {n}-token chunk at k={k}, all {wl.layers} "
                "layers per call (RoPE at the extraction positions, SIF-masked attention); "
                "L2 flushed before each call (untimed)",
        "kernel_ms": round(kernel_ms, 5) if kernel_ms else None,
        "roofline": {"bound": "tensor" if tensor else "hbm",
                     "kernel": "extraction call (extract_rope_kernel, attn_tc_kernel x2)",
                     "achieved": round(tfs, 2) if tensor else round(gbs, 1),
                     "peak": bf16 if tensor else hbm, "unit": "TFLOP/s" if tensor else "GB/s",
                     "frac": round(tfs / bf16 if tensor else gbs / hbm, 4),
                     "peak_source": f"{src} " + ("bf16_tflops (burst)" if tensor else "hbm_gbs"),
                     "flops_per_launch": flops, "bytes_per_launch": nbytes,
                     "traffic": captured_traffic("extract_call", wl.name),
                     "tensor_frac": round(tfs / bf16, 4), "hbm_frac": round(gbs / hbm, 4)},
    }


def decode_on_tensor_cores(wl, keys_per_request, sms=152):
    """The decode route c2kv_decode takes for this shape (its rule: the tensor-core kernel for
    bf16 at head_dim 128 when the (layer, request, KV head) units fit in one wave of SMs or a
    request has at least 32 key tiles; the CUDA-core kernel otherwise)."""
    units = wl.layers * wl.batch * wl.n_kv_heads
    return wl.dtype == "bf16" and wl.head_dim == 128 and (units <= sms or keys_per_request >= 32 * 128)


def decode_line(wl, world, dec_ms, dec_kernel_ms, dec_keys, hbm, src):
    eb = 4 if wl.dtype == "f32" else 2
    bytes_step = dec_keys * wl.layers * wl.n_kv_heads * wl.head_dim * eb * 2
    kernel_gbs = bytes_step / (dec_kernel_ms / 1e3) / 1e9 if dec_kernel_ms else None
    tc = decode_on_tensor_cores(wl, dec_keys / wl.batch)
    kernel = ("attn_tc_decode_kernel (one-row suffix; key tiles split between the two softmax "
              "warpgroups; splits merged in the kernel)") if tc else "decode_kernel (+ merge)"
    return {
        "metric": "decode tokens/s", "unit": "tokens/s",
        "value": round(wl.batch * world / (dec_ms / 1e3), 1),
        "ms_per_step": round(dec_ms, 5),
        "what": "one new token per request after the suffix, all layers per call (c2kv_decode); "
                "RoPE/append and the split-KV attention; L2 flushed before each step (untimed)",
        "keys_per_request": round(dec_keys / wl.batch, 1),
        "kernel_ms": round(dec_kernel_ms, 5),
        "roofline": {"bound": "hbm", "kernel": kernel,
                     "achieved": round(kernel_gbs, 1) if kernel_gbs else None, "peak": hbm,
                     "unit": "GB/s", "frac": round(kernel_gbs / hbm, 4) if kernel_gbs else None,
                     "peak_source": f"{src} hbm_gbs", "bytes_per_launch": int(bytes_step),
                     "traffic": captured_traffic("attn_tc_decode_kernel" if tc else "decode_kernel",
                                                 wl.name)},
    }


def long_decode(torch, c2kv, hbm, src, flush, keys=131072, steps=5, warmup=3):
    """Decode at the top of the paper's 16k-128k context range: one request whose composed
    cache holds `keys` slots (64 chunks x 2048 tokens at k = 1, Llama-3-8B layer shape, one
    layer), its stored slots drawn on the device; `steps` timed decode steps after a short
    suffix, L2 flushed before each; the kernel from the library's trace against HBM."""
    base = synth.workload("sweep_k1")
    chunks = keys // base.chunk_tokens
    wl = synth.scaled(base, layers=1, batch=1, chunks_per_request=chunks, pool_chunks=chunks,
                      n_suffix=4)
    stream = torch.cuda.current_stream()
    m = wl.chunk_tokens
    ctx = c2kv.c2kv_create(1, wl.n_q_heads, wl.n_kv_heads, wl.head_dim, wl.rope_theta,
                           c2kv.DTYPE_BF16, pool_slots=chunks * m + 64, stream=stream)
    try:
        gen = torch.Generator(device="cuda").manual_seed(7)
        shape = (1, m, wl.n_kv_heads, wl.head_dim)
        ids = []
        for _ in range(chunks):
            kd = torch.randn(shape, device="cuda", generator=gen).to(torch.bfloat16)
            vd = torch.randn(shape, device="cuda", generator=gen).to(torch.bfloat16)
            ids.append(c2kv.c2kv_compress_chunk(ctx, kd, vd, wl.chunk_tokens, 1, c2kv.MODE_STORED))
        q_dev = [torch.randn((1, 1, wl.n_suffix, h, wl.head_dim), device="cuda", generator=gen)
                 .to(torch.bfloat16) for h in (wl.n_q_heads, wl.n_kv_heads, wl.n_kv_heads)]
        out = torch.empty_like(q_dev[0])
        events = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(steps)]
        ms, kern_ms, kv, per = decode_measure(c2kv, torch, ctx, wl, stream, np.array([0, chunks], np.int32),
                                              ids, None, q_dev, out, steps, warmup, events, flush)
        line = decode_line(wl, 1, statistics.median(per), kern_ms, kv, hbm, src)
        line["what"] = (f"one request over a composed cache of {keys} keys (the paper's 16k-128k "
                        "decode range), Llama-3-8B layer shape, one layer; " + line["what"])
        line["roofline"]["traffic"] = captured_traffic("attn_tc_decode_kernel", "decode_long")
        return line
    finally:
        c2kv.c2kv_destroy(ctx)


# --------------------------------------------------------------------------- other workloads

SIDE_WORKLOADS = ("tiny_f32", "batched", "long70b", "sweep_k1", "sweep_k4", "sweep_k8", "sweep_k10",
                  "sweep_k16")

# The fp32 path's attention runs on the CUDA cores: its peak is derived, not measured, from
# 128 FP32 lanes per SM x 2 flops per FMA x 152 SMs x the 2.07 GHz maximum SM clock.
FP32_ALU_TFLOPS = 128 * 2 * 152 * 2.07e9 / 1e12


def error_vs_oracle(got, ref, tol):
    """max |gpu - oracle|, the largest relative error over elements whose oracle magnitude
    is at least the tolerance (below it the absolute term of the bound governs), and the
    largest ratio of the error to the element's bound tol + tol * |oracle| (parity: <= 1)."""
    diff = np.abs(got - ref)
    big = np.abs(ref) >= tol
    return {"max_abs": float(diff.max()),
            "max_rel": float((diff[big] / np.abs(ref[big])).max()) if big.any() else 0.0,
            "tol_ratio": round(float((diff / (tol + tol * np.abs(ref))).max()), 4),
            "tol": tol}


def side_workload(name, steps, warmup, torch, c2kv, hbm, bf16, src, flush, with_oracle=True):
    """One of the other workloads at full size on one GPU, through c2kv_compose_attend as the
    headline step: the step time (median of `steps`, L2 flushed before each), the compose
    kernel against HBM (cold, and warm: right after an identical compose, inputs in L2 where
    they fit), the attention kernel against the bf16 tensor peak, a decode step after the
    suffix, and the output error against the oracle on one sampled (layer, request).

    The chunks of the sampled request (request 0) are synth's, so that the oracle sees the
    same bits; the pool's other chunks are drawn on the device with the same shape and
    outlier channels (their values do not change the timing)."""
    wl = synth.workload(name)
    f = workload_facts(wl)
    tdt = torch.float32 if wl.dtype == "f32" else torch.bfloat16
    E = torch.cuda.Event
    stream = torch.cuda.current_stream()
    reqs = synth.requests(wl, 0)
    m = f["slots_per_chunk"]
    pool_ids = sorted({c for ids, _ in reqs for c in ids})
    t_setup = time.perf_counter()
    ctx = c2kv.c2kv_create(wl.layers, wl.n_q_heads, wl.n_kv_heads, wl.head_dim, wl.rope_theta,
                           c2kv.DTYPE_F32 if wl.dtype == "f32" else c2kv.DTYPE_BF16,
                           pool_slots=len(pool_ids) * m + 64, stream=stream)
    try:
        sample = reqs[0]
        mult = torch.from_numpy(synth.outlier_mask(wl, 0)).to("cuda")
        gen = torch.Generator(device="cuda").manual_seed(3)
        shape = (wl.layers, m, wl.n_kv_heads, wl.head_dim)
        dev, oracle_chunks = {}, {}
        for cid in pool_ids:
            if cid in sample[0]:
                ks, vs = synth.chunk_slots(wl, cid, m, 0)
                kd, vd = (torch.from_numpy(x).to("cuda", tdt) for x in (ks, vs))
                oracle_chunks[cid] = (ks[:1].astype(np.float64), vs[:1].astype(np.float64),
                                      wl.chunk_tokens, wl.ratio_k)
            else:
                kd = (torch.randn(shape, device="cuda", generator=gen) * mult).to(tdt)
                vd = (torch.randn(shape, device="cuda", generator=gen) * mult).to(tdt)
            dev[cid] = c2kv.c2kv_compress_chunk(ctx, kd, vd, wl.chunk_tokens, wl.ratio_k,
                                                c2kv.MODE_STORED)
        req_ptr = np.cumsum([0] + [len(ids) for ids, _ in reqs]).astype(np.int32)
        ids = [dev[c] for ids_, _ in reqs for c in ids_]
        positions = [o for _, offs in reqs for o in offs]
        qn, kn, vn = synth.suffix(wl, 0)
        q_dev = [torch.from_numpy(x).to("cuda", tdt) for x in (qn, kn, vn)]
        out = torch.empty_like(q_dev[0])
        c2kv.c2kv_sync(ctx)
        setup_s = time.perf_counter() - t_setup

        def step():
            cache = c2kv.c2kv_compose_attend(ctx, req_ptr, ids, positions, wl.n_suffix, *q_dev,
                                             wl.n_suffix, out)
            c2kv.c2kv_cache_release(ctx, cache)

        def timed(fn, cold):
            evs = [(E(enable_timing=True), E(enable_timing=True)) for _ in range(steps)]
            for a, b in evs:
                if cold:
                    flush()
                else:
                    fn()                       # the identical call just before: inputs in L2
                a.record(stream)
                fn()
                b.record(stream)
            torch.cuda.synchronize()
            return statistics.median(x.elapsed_time(y) for x, y in evs)

        def compose_only():
            c2kv.c2kv_cache_release(ctx, c2kv.c2kv_compose(ctx, req_ptr, ids, positions, wl.n_suffix))

        for _ in range(warmup):
            flush()
            step()
            compose_only()
        c2kv.c2kv_sync(ctx)
        step_ms = timed(step, cold=True)
        compose_cold_ms = timed(compose_only, cold=True)
        compose_warm_ms = timed(compose_only, cold=False)
        c2kv.c2kv_profile_read(ctx)
        c2kv.c2kv_profile_enable(ctx, True)
        for _ in range(steps):
            flush()
            step()
        kern = c2kv.c2kv_profile_read(ctx)
        c2kv.c2kv_profile_enable(ctx, False)
        c2kv.c2kv_sync(ctx)
        fused = kern["fused"][1] > 0
        kc = kern["compose"][0]
        ka = kern["attention"][0] + kern["combine"][0]
        entry = {
            "workload": describe(wl),
            "step_ms": round(step_ms, 5),
            "composed_tokens_per_s": round(f["positions"] / (step_ms / 1e3), 1),
            "route": "fused compose + attention kernel" if fused else
                     "compose, then attention (suffix kernel beside compose)",
        }
        if fused:
            entry["fused"] = fused_roofline(kern["fused"][0], f, hbm, bf16, src)
        else:
            comp_gbs = f["compose_bytes"] / (kc / 1e3) / 1e9
            warm_gbs = f["compose_bytes"] / (compose_warm_ms / 1e3) / 1e9
            attn_tfs = f["attn_flops"] / (ka / 1e3) / 1e12
            attn_gbs = f["attn_bytes"] / (ka / 1e3) / 1e9
            entry["compose"] = {
                "kernel_ms": round(kc, 5), "achieved_gbs": round(comp_gbs, 1),
                "frac": round(comp_gbs / hbm, 4), "peak": hbm, "peak_source": f"{src} hbm_gbs",
                "bytes_per_launch": f["compose_bytes"],
                "cold_call_ms": round(compose_cold_ms, 5), "warm_call_ms": round(compose_warm_ms, 5),
                "warm_gbs": round(warm_gbs, 1),
                "traffic": captured_traffic("compose_kernel", name)}
            if len(pool_ids) < len(ids):
                # repeated chunks (Zipf draws): each distinct chunk's slots read once, every
                # composed row written; reads of repeats can hit L2, so the algorithmic rate
                # above may exceed HBM's
                reads = wl.layers * wl.batch * f["slots"] * f["row_bytes"] * 2
                uniq = wl.layers * len(pool_ids) * m * f["row_bytes"] * 2 + (f["compose_bytes"] - reads)
                entry["compose"]["unique_chunk_bytes"] = uniq
                entry["compose"]["unique_chunk_gbs"] = round(uniq / (kc / 1e3) / 1e9, 1)
            entry["suffix_kernel_ms"] = round(kern["suffix"][0], 5)
            if wl.dtype == "f32":     # CUDA-core kernel: against the FP32 FMA rate
                entry["attention"] = {
                    "kernel": "attn_simt_kernel", "bound": "alu",
                    "kernel_ms": round(ka, 5), "achieved_tflops": round(attn_tfs, 4),
                    "frac": round(attn_tfs / FP32_ALU_TFLOPS, 5), "peak": round(FP32_ALU_TFLOPS, 1),
                    "peak_source": "derived: 128 FP32 lanes x 2 flop x 152 SMs x 2.07 GHz",
                    "flops_per_launch": f["attn_flops"], "hbm_frac": round(attn_gbs / hbm, 5)}
            else:
                entry["attention"] = {
                    "kernel_ms": round(ka, 5), "achieved_tflops": round(attn_tfs, 2),
                    "frac": round(attn_tfs / bf16, 4), "peak": bf16,
                    "peak_source": f"{src} bf16_tflops (burst)", "flops_per_launch": f["attn_flops"],
                    "hbm_frac": round(attn_gbs / hbm, 4),
                    "split_merge_ms": round(kern["combine"][0], 5),
                    "traffic": captured_traffic("attn_tc_kernel", name)}
        # decode after the suffix, at this workload's context length
        dec_events = [[E(enable_timing=True) for _ in range(2)] for _ in range(steps)]
        d_ms, d_kern, d_keys, d_per = decode_measure(c2kv, torch, ctx, wl, stream, req_ptr, ids,
                                                      positions, q_dev, out, steps, warmup,
                                                      dec_events, flush)
        dline = decode_line(wl, 1, statistics.median(d_per), d_kern, d_keys, hbm, src)
        entry["decode"] = {k: dline[k] for k in ("value", "unit", "ms_per_step", "keys_per_request",
                                                 "kernel_ms")}
        entry["decode"]["roofline"] = {k: dline["roofline"][k] for k in ("achieved", "frac", "unit",
                                                                         "bytes_per_launch", "traffic")}
        # output error against the oracle: layer 0 of request 0, every suffix row and head
        if with_oracle:
            cache = c2kv.c2kv_compose_attend(ctx, req_ptr, ids, positions, wl.n_suffix, *q_dev,
                                             wl.n_suffix, out)
            c2kv.c2kv_sync(ctx)
            got = out[0, 0].double().cpu().numpy()
            c2kv.c2kv_cache_release(ctx, cache)
            from oracle import c2kv_oracle as orc
            t0 = time.perf_counter()
            ref = orc.run_request(oracle_chunks, sample[0], sample[1], qn[:1, 0], kn[:1, 0],
                                  vn[:1, 0], wl.rope_theta, wl.dtype)
            tol = 1e-5 if wl.dtype == "f32" else 2e-2
            entry["error_vs_oracle"] = dict(error_vs_oracle(got, ref["out"][0], tol),
                                            sample=f"layer 0 of request 0: {wl.n_suffix} suffix "
                                                   f"tokens x {wl.n_q_heads} heads x {wl.head_dim}",
                                            oracle_s=round(time.perf_counter() - t0, 2))
        entry["setup_s"] = round(setup_s, 2)
        return entry
    finally:
        c2kv.c2kv_destroy(ctx)


def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def run_ours(args):
    import torch
    import __graft_entry__ as g
    g.build()
    from paper_2607_17715_gb300 import c2kv

    world, rank, local = dist_setup()
    torch.cuda.set_device(local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    wl = synth.workload(args.workload)
    arm = Arm(wl, rank, world, torch=torch, c2kv=c2kv, attn_split=args.attn_split)
    f = arm.facts
    E = torch.cuda.Event

    def barrier():
        torch.cuda.synchronize()
        if world > 1:
            torch.distributed.barrier()
            torch.cuda.synchronize()

    for _ in range(args.warmup):
        arm.flush_l2()
        arm.step_device([E(enable_timing=True) for _ in range(4)])
        arm.flush_l2()
        arm.step_device([E(enable_timing=True) for _ in range(4)], fused=False)
    c2kv.c2kv_sync(arm.ctx)

    events = [[E(enable_timing=True) for _ in range(4)] for _ in range(args.steps)]
    barrier()
    with ClockSampler(local) as clocks:
        for _ in range(2):           # the GPU idled while the sampler started: bring it back up
            arm.flush_l2()
            arm.step_device([E(enable_timing=True) for _ in range(4)])
        barrier()
        t0 = time.perf_counter()
        for i in range(args.steps):
            arm.flush_l2()           # untimed: L2 holds none of this step's inputs
            arm.step_device(events[i])
        torch.cuda.synchronize()
        wall = time.perf_counter() - t0
    barrier()
    c2kv.c2kv_sync(arm.ctx)
    # Per-kernel device times: the same steps again with the library's trace on (events on
    # its stream around every launch).  An event recorded between two kernels holds the
    # second back by a few us, so the steps that give the headline run without the trace.
    def traced(fused):
        c2kv.c2kv_profile_read(arm.ctx)        # drop anything recorded before
        c2kv.c2kv_profile_enable(arm.ctx, True)
        evs = [[E(enable_timing=True) for _ in range(4)] for _ in range(args.steps)]
        for i in range(args.steps):
            arm.flush_l2()
            arm.step_device(evs[i], fused=fused)
        torch.cuda.synchronize()
        c2kv.c2kv_sync(arm.ctx)
        k = c2kv.c2kv_profile_read(arm.ctx)    # mean device ms per kernel kind
        c2kv.c2kv_profile_enable(arm.ctx, False)
        return k
    kern = traced(True)
    step_ms = [ev[0].elapsed_time(ev[3]) for ev in events]
    total_ms = sum(step_ms)
    # the same steps as separate compose and attend calls: the two kernels the fused path
    # replaces, each against its own roofline
    un_events = [[E(enable_timing=True) for _ in range(4)] for _ in range(args.steps)]
    barrier()
    for i in range(args.steps):
        arm.flush_l2()
        arm.step_device(un_events[i], fused=False)
    torch.cuda.synchronize()
    c2kv.c2kv_sync(arm.ctx)
    un_total_ms = sum(ev[0].elapsed_time(ev[3]) for ev in un_events)
    compose_ms = [ev[0].elapsed_time(ev[1]) for ev in un_events]
    attend_ms = [ev[1].elapsed_time(ev[2]) for ev in un_events]
    kern_un = traced(False)
    compose_warm_ms = arm.compose_warm(args.steps)

    # end to end from host buffers (host->device traffic inside the timed region), both
    # ways the library offers: zero-copy compose from pinned host slots, and staged copies
    def timed_e2e(step):
        # the first passes over pinned host memory are slower (page walks over the link):
        # as many warm-up steps as the device step gets
        for _ in range(max(3, args.warmup)):
            step()
        barrier()
        e0, e1 = E(enable_timing=True), E(enable_timing=True)
        e0.record(arm.stream)
        for _ in range(args.steps):
            step()
        e1.record(arm.stream)
        torch.cuda.synchronize()
        c2kv.c2kv_sync(arm.ctx)
        return e0.elapsed_time(e1)

    e2e_ms = timed_e2e(arm.step_e2e_host)
    staged_ms = timed_e2e(arm.step_e2e)
    h2d, d2h = arm.e2e_bytes(zero_copy=True)
    h2d_staged, _ = arm.e2e_bytes(zero_copy=False)

    # decode after the suffix (one new token per request per step, all layers)
    dec_events = [[E(enable_timing=True) for _ in range(2)] for _ in range(args.steps)]
    dec_ms, dec_kernel_ms, dec_keys, _ = arm.decode_run(args.steps, args.warmup, dec_events)

    # extraction attention over one chunk (the encoding side, Sec. 3.3)
    ext_events = [[E(enable_timing=True) for _ in range(2)] for _ in range(args.steps)]
    ext_ms, ext_kernel_ms = arm.extract_run(args.steps, args.warmup, ext_events)

    from paper_2607_17715_gb300.shard import max_over_ranks
    total_ms, un_total_ms, e2e_ms, staged_ms, dec_ms, ext_ms = max_over_ranks(
        [total_ms, un_total_ms, e2e_ms, staged_ms, dec_ms, ext_ms], device="cuda")
    arm.close()
    hbm, bf16, bf16_sus, src = measured_peaks()
    # the other workloads at full size, each on this rank's GPU (requests sharded like the
    # headline would take a global batch; here every rank runs its own replica)
    workloads = {}
    if args.workloads and rank == 0:
        for name in args.workloads.split(","):
            workloads[name] = side_workload(name, args.side_steps, args.warmup, torch, c2kv, hbm, bf16,
                                            src, arm.flush_l2, with_oracle=not args.no_cpu_baseline)
    if rank != 0:
        if world > 1:
            torch.distributed.destroy_process_group()
        return

    gf = workload_facts(synth.scaled(wl, batch=wl.batch * world))   # whole job
    positions = gf["positions"] * args.steps
    value = positions / (total_ms / 1e3)
    c_ms = statistics.mean(compose_ms)
    a_ms = statistics.mean(attend_ms)
    kc_ms = kern_un["compose"][0] or c_ms      # compose kernel alone (library events)
    # attention kernel (plus the merge of its key-range splits, when it was split)
    ka_ms = (kern_un["attention"][0] + kern_un["combine"][0]) or a_ms
    fused_ran = kern["fused"][1] > 0
    step_kernels = {k: round(v[0], 5) for k, v in kern.items() if v[1]}
    comp_gbs = f["compose_bytes"] / (kc_ms / 1e3) / 1e9
    attn_tfs = f["attn_flops"] / (ka_ms / 1e3) / 1e12
    clk = clocks.summary()
    line = {
        "metric": METRIC, "value": round(value, 1), "unit": "tokens/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(total_ms / args.steps, 5),
        "ms_per_step_median": round(statistics.median(step_ms), 5), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": wl.dtype, "data": "synthetic",
        "config": job_config(wl, world),
        "parallelism": f"dp{world}: requests sharded over ranks, no data-path collective",
        "l2": "flushed between timed steps (256 MB write, untimed)",
        "detail": {"ttft_proxy_ms_per_layer": round(kc_ms / wl.layers, 6),
                   "step": ("c2kv_compose_attend: one kernel (compose, suffix preparation and "
                            "attention fused)" if fused_ran
                            else "c2kv_compose_attend: compose, then attention"),
                   "kernel_ms": step_kernels,
                   "unfused": {"value": round(positions / (un_total_ms / 1e3), 1),
                               "ms_per_step": round(un_total_ms / args.steps, 5),
                               "compose_call_ms": round(c_ms, 5), "attend_call_ms": round(a_ms, 5),
                               "compose_call_ms_median": round(statistics.median(compose_ms), 5),
                               "compose_warm_call_ms": round(compose_warm_ms, 5),
                               "compose_warm_gbs": round(f["compose_bytes"] / (compose_warm_ms / 1e3) / 1e9, 1),
                               "kernel_ms": {k: round(v[0], 5) for k, v in kern_un.items() if v[1]}},
                   "compose_gbs": round(comp_gbs, 1), "attend_tflops": round(attn_tfs, 2),
                   "compose_bytes": f["compose_bytes"], "attend_flops": f["attn_flops"],
                   "fused_bytes": f["fused_bytes"], "wall_s": round(wall, 4)},
        # the dominant kernel of the step (by device time) carries "roofline"; the separate
        # compose and attention kernels (from the same steps run as separate calls) are
        # reported beside it.  Attention is HBM- or tensor-bound depending on its arithmetic
        # intensity relative to the ridge of the measured peaks.
        **step_rooflines(fused_ran, kern, kc_ms, ka_ms, f, hbm, bf16, src),
        "e2e": {"value": round(positions / (e2e_ms / 1e3), 1),
                "unit": "tokens/s", "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                "ms_per_step": round(e2e_ms / args.steps, 4),
                "path": "chunks (MODE_HOST) read by compose across the CPU-GPU link; suffix Q/K/V "
                        "and output in pinned host memory, copied in and out by the call per layer group",
                "staged": {"value": round(positions / (staged_ms / 1e3), 1),
                           "ms_per_step": round(staged_ms / args.steps, 4),
                           "h2d_bytes_per_step": h2d_staged,
                           "path": "chunks copied host->pool (MODE_STORED) and the suffix "
                                   "copied in, then one call (fused on this route), output "
                                   "copied back"}},
        # decode after the suffix: tokens generated per second over the whole job, and the
        # decode kernel against HBM (algorithmic bytes: K and V of every key it attends to)
        "decode": decode_line(wl, world, dec_ms, dec_kernel_ms, dec_keys, hbm, src),
        # extraction attention (the C2 Extractor's masked attention) over one chunk
        "extract": extract_line(wl, world, ext_ms, ext_kernel_ms, hbm, bf16, src),
        # every kernel the library launched in the timed steps (counted by its trace of the
        # identical traced pass; a fused record covers two launches, the suffix angles kernel
        # and the fused kernel)
        "gpu_launches": sum(v[1] for v in kern.values()) + kern.get("fused", (0.0, 0))[1],
        "clocks": clk,
    }
    if not args.no_long_decode:
        # decode over a 128k-key composed cache (one layer)
        line["decode_long"] = long_decode(torch, c2kv, hbm, src, arm.flush_l2)
    if workloads:
        # configs 3-5 (batched reuse, long context, the compression-ratio sweep with its
        # uncompressed control), each run once at full size in the same process
        line["workloads"] = workloads
    if not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(wl, budget_s=args.cpu_budget)
    print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()


# --------------------------------------------------------------------------- oracle arm

def cpu_threads():
    try:
        from threadpoolctl import threadpool_info
        n = [i["num_threads"] for i in threadpool_info() if i.get("user_api") == "blas"]
        if n:
            return max(n)
    except Exception:
        pass
    return len(os.sched_getaffinity(0))


def cpu_model():
    """The host CPU as /proc/cpuinfo names it (x86: model name; Arm: implementer and part)."""
    import platform
    try:
        with open("/proc/cpuinfo") as fh:
            info = fh.read()
    except OSError:
        return platform.machine()
    for line in info.splitlines():
        if line.lower().startswith("model name"):
            return line.split(":", 1)[1].strip()
    fields = {}
    for line in info.splitlines():
        if ":" in line:
            k, v = (x.strip() for x in line.split(":", 1))
            fields.setdefault(k, v)
    if "CPU part" in fields:
        return f"{platform.machine()}, CPU implementer {fields.get('CPU implementer', '?')}, part {fields['CPU part']}"
    return platform.machine()


def oracle_sample(wl, layers, seed=0):
    """Time the oracle's compose + attend for `layers` layers of request 0's workload."""
    from oracle import c2kv_oracle as orc
    sub = synth.scaled(wl, layers=1)
    reqs = synth.requests(wl, seed)
    m = -(-wl.chunk_tokens // wl.ratio_k)
    ids, offs = reqs[0]
    chunks = {}
    for cid in sorted(set(ids)):
        ks, vs = synth.chunk_slots(sub, cid, m, seed)
        chunks[cid] = (ks.astype(np.float64), vs.astype(np.float64), wl.chunk_tokens,
                       wl.ratio_k)
    q, k, v = synth.suffix(sub, seed)
    t0 = time.perf_counter()
    for _ in range(layers):
        orc.run_request(chunks, ids, offs, q[:, 0], k[:, 0], v[:, 0], wl.rope_theta, wl.dtype)
    return time.perf_counter() - t0


def oracle_sample_one_core(wl, layers):
    """oracle_sample in a child process confined to one core with single-threaded BLAS
    (the thread pools are sized when numpy loads, so it takes a fresh interpreter)."""
    code = (f"import os, sys\n"
            f"os.sched_setaffinity(0, {{sorted(os.sched_getaffinity(0))[0]}})\n"
            f"sys.path.insert(0, {ROOT!r})\n"
            f"import bench, synth\n"
            f"print('SECONDS', bench.oracle_sample(synth.workload({wl.name!r}), {layers}))\n")
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1")
    res = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True,
                         timeout=600)
    for line in res.stdout.splitlines():
        if line.startswith("SECONDS"):
            return float(line.split()[1])
    return None


def cpu_baseline(wl, budget_s=15.0, one_core_budget_s=8.0):
    """The oracle as it stands on this host's cores, on a bounded sample: as many layers of
    request 0 as fit in about `budget_s` seconds, scaled to the whole batch; and the same on
    one core."""
    f = workload_facts(wl)
    t1 = oracle_sample(wl, 1)
    n = int(max(1, min(wl.layers * wl.batch, budget_s // max(t1, 1e-3))))
    t = oracle_sample(wl, n)
    per_layer_req = t / n
    step_s = per_layer_req * wl.layers * wl.batch
    out = {"value": round(f["positions"] / step_s, 1), "unit": "tokens/s",
           "cores": cpu_threads(), "cpu": cpu_model(), "kind": "oracle",
           "sample": f"{n} (layer, request) compose+attend passes of the oracle (fp64 numpy), "
                     f"{t:.1f} s, scaled to {wl.layers} layers x {wl.batch} requests"}
    # one core: as many passes as fit in about one_core_budget_s at the all-core rate x 4
    n1 = int(max(1, min(wl.layers * wl.batch, one_core_budget_s // max(4 * per_layer_req, 1e-3))))
    t1c = oracle_sample_one_core(wl, n1)
    if t1c:
        out["one_core"] = {"value": round(f["positions"] / (t1c / n1 * wl.layers * wl.batch), 1),
                           "cores": 1,
                           "sample": f"{n1} (layer, request) passes, {t1c:.1f} s, in a child "
                                     "process pinned to one core with single-threaded BLAS"}
    return out


def job_config(wl, world):
    """The workload a line describes: the same object in both arms' lines."""
    return {"workload": describe(wl), "global_batch": wl.batch * world}


def run_reference(args):
    """The oracle arm.  Each step is one bounded sample of the workload: compose + attend of
    one layer of request 0, i.e. 1 / (layers * requests) of the whole step; ms_per_step is
    that sample's measured time, and value is the same metric (composed positions of the
    whole job per second) at the sample's rate."""
    world, rank, _ = dist_setup()
    if rank != 0:
        return
    wl = synth.workload(args.workload)
    f = workload_facts(synth.scaled(wl, batch=wl.batch * world))
    for _ in range(args.warmup):
        oracle_sample(wl, 1)
    times = [oracle_sample(wl, 1) for _ in range(args.steps)]
    share = wl.layers * wl.batch * world                 # samples in one whole step
    sample_s = statistics.mean(times)
    value = f["positions"] / share / sample_s
    cores = cpu_threads()
    line = {
        "impl": "reference", "metric": METRIC, "value": round(value, 1), "unit": "tokens/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(sample_s * 1e3, 3),
        "ms_per_step_median": round(statistics.median(times) * 1e3, 3),
        "step": f"one sample: compose + attend of 1 layer of request 0 (1/{share} of a whole "
                f"step of the workload)",
        "ms_per_whole_step_extrapolated": round(sample_s * share * 1e3, 3),
        "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": job_config(wl, world),
        "parallelism": "cpu oracle (rank 0 only)",
        "cpu_baseline": {"value": round(value, 1), "unit": "tokens/s", "cores": cores,
                         "kind": "oracle",
                         "sample": f"each step: compose+attend of 1 layer of request 0 "
                                   f"(1/{share} of the workload's step)"},
        "e2e": {"value": round(value, 1), "unit": "tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="llama8b", choices=sorted(synth.WORKLOADS))
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-long-decode", action="store_true",
                    help="skip the decode leg over a 128k-key cache")
    ap.add_argument("--cpu-budget", type=float, default=15.0)
    ap.add_argument("--attn-split", type=int, default=0,
                    help="key-range splits of the attention (0 = library's choice)")
    ap.add_argument("--workloads", default=",".join(SIDE_WORKLOADS),
                    help="other workloads measured after the headline ('' = none)")
    ap.add_argument("--side-steps", type=int, default=10,
                    help="timed steps of each other workload (median reported)")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
