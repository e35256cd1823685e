"""Data-parallel placement of independent requests over ranks (one GPU per rank).

Requests share nothing on this path -- each composes its own cache and attends over it --
so a batch splits across ranks with no data-path collective: rank r takes a contiguous
share of the global request list.  Only timing crosses ranks (max over ranks).
"""
from __future__ import annotations


def shard_range(n_items: int, rank: int, world: int) -> tuple[int, int]:
    """Contiguous [start, end) share of n_items for `rank` of `world`; shares differ by at
    most one item and cover every item exactly once."""
    if world < 1 or not 0 <= rank < world or n_items < 0:
        raise ValueError("bad shard arguments")
    base, extra = divmod(n_items, world)
    start = rank * base + min(rank, extra)
    return start, start + base + (1 if rank < extra else 0)


def max_over_ranks(values, device=None):
    """Element-wise max of a list of floats over all ranks (identity without a process
    group).  Works on any torch.distributed backend (gloo on CPU, nccl on GPU)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return list(values)
    t = torch.tensor(list(values), dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return t.tolist()
