"""Multi-rank host logic on CPU with the gloo backend (world_size 2): request sharding
covers the batch exactly once, the max-over-ranks timing reduction, and per-rank results
(the oracle run on each rank's share) reassemble into the unsharded result."""
import os
import socket

import numpy as np
import pytest
import torch.multiprocessing as mp

from paper_2607_17715_gb300.shard import shard_range


@pytest.mark.parametrize("n,world", [(1, 1), (5, 2), (16, 4), (3, 8), (0, 2), (7, 3)])
def test_shard_range_partitions(n, world):
    seen = []
    for r in range(world):
        a, b = shard_range(n, r, world)
        assert 0 <= a <= b <= n and b - a in (n // world, n // world + 1)
        seen.extend(range(a, b))
    assert seen == list(range(n))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out_dir):
    import torch.distributed as dist

    import synth
    from oracle import c2kv_oracle as orc
    from paper_2607_17715_gb300.shard import max_over_ranks, shard_range

    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    wl = synth.scaled(synth.workload("tiny_f32"), batch=3, pool_chunks=4, chunks_per_request=2,
                      draw="distinct", chunk_tokens=40, n_suffix=5, n_q_heads=2, n_kv_heads=1,
                      head_dim=64)
    reqs = synth.requests(wl)
    q, k, v = synth.suffix(wl)
    a, b = shard_range(len(reqs), rank, world)
    mine = {}
    for r in range(a, b):
        ids, offs = reqs[r]
        chunks = {}
        for cid in ids:
            kt, vt = synth.chunk_tokens(wl, cid)
            chunks[cid] = orc.compress_chunk(kt, vt, wl.chunk_tokens, wl.ratio_k,
                                             wl.rope_theta, wl.dtype, "meanpool") + (
                wl.chunk_tokens, wl.ratio_k)
        mine[r] = orc.run_request(chunks, ids, offs, q[:, r], k[:, r], v[:, r],
                                  wl.rope_theta, wl.dtype)["out"]
    gathered = [None] * world
    dist.all_gather_object(gathered, mine)
    worst = max_over_ranks([float(rank + 1), -float(rank)])
    if rank == 0:
        merged = {}
        for part in gathered:
            merged.update(part)
        np.savez(os.path.join(out_dir, "merged.npz"),
                 **{str(r): merged[r] for r in sorted(merged)}, worst=np.array(worst))
    dist.barrier()
    dist.destroy_process_group()


def test_gloo_two_ranks_reassemble(tmp_path):
    world = 2
    mp.start_processes(_worker, args=(world, _free_port(), str(tmp_path)), nprocs=world,
                       join=True, start_method="spawn")
    got = np.load(tmp_path / "merged.npz")
    assert list(got["worst"]) == [2.0, 0.0]              # max over ranks of (rank+1, -rank)
    import synth
    from oracle import c2kv_oracle as orc
    wl = synth.scaled(synth.workload("tiny_f32"), batch=3, pool_chunks=4, chunks_per_request=2,
                      draw="distinct", chunk_tokens=40, n_suffix=5, n_q_heads=2, n_kv_heads=1,
                      head_dim=64)
    reqs = synth.requests(wl)
    q, k, v = synth.suffix(wl)
    for r, (ids, offs) in enumerate(reqs):
        chunks = {}
        for cid in ids:
            kt, vt = synth.chunk_tokens(wl, cid)
            chunks[cid] = orc.compress_chunk(kt, vt, wl.chunk_tokens, wl.ratio_k,
                                             wl.rope_theta, wl.dtype, "meanpool") + (
                wl.chunk_tokens, wl.ratio_k)
        ref = orc.run_request(chunks, ids, offs, q[:, r], k[:, r], v[:, r], wl.rope_theta,
                              wl.dtype)["out"]
        assert np.array_equal(got[str(r)], ref)
