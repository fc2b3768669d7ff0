"""Splitting one search, or one batch of searches, over several ranks (one GPU each).

The mapping index space [0, 3^n) splits into contiguous ranges; each rank
searches its own with ``bf_search_range`` and the ranks exchange one packed
key each (makespan << 32 | index).  The smallest key is the answer of the
whole search: ranges compose because the argmin is a minimum over (makespan,
index) pairs.  The exchange is the only collective, 8 bytes per rank.

A batch of independent scenarios splits into contiguous blocks of scenarios,
one per rank (``bf_search_batch`` on each); one all-gather of the per-rank
result lists returns every scenario's optimum to every rank.
"""
from __future__ import annotations

from typing import Callable, List, Optional, Sequence, Tuple

INFEASIBLE = 0xFFFFFFFF
NO_KEY = (1 << 64) - 1


def shard_range(total: int, rank: int, world: int) -> Tuple[int, int]:
    """(first, count) of rank `rank`'s contiguous share of [0, total)."""
    lo = total * rank // world
    hi = total * (rank + 1) // world
    return lo, hi - lo


def pack_key(index: int, makespan: int, feasible: bool) -> int:
    return (makespan << 32) | index if feasible else NO_KEY


def unpack_key(key: int) -> Tuple[int, int, bool]:
    """(index, makespan, feasible)."""
    if key == NO_KEY or (key >> 32) == INFEASIBLE:
        return -1, INFEASIBLE, False
    return key & 0xFFFFFFFF, key >> 32, True


def min_key_over_ranks(key: int, group=None) -> int:
    """Smallest packed key over all ranks of `group` (one all-gather of 8 bytes per rank)."""
    import torch
    import torch.distributed as dist
    world = dist.get_world_size(group)
    backend = dist.get_backend(group)
    device = "cuda" if backend == "nccl" else "cpu"
    # int64 holds the key's bit pattern; compare as unsigned on the host.
    mine = torch.tensor([key - (1 << 64) if key >= (1 << 63) else key], dtype=torch.int64, device=device)
    parts = [torch.empty_like(mine) for _ in range(world)]
    dist.all_gather(parts, mine, group=group)
    return min(int(p.item()) & ((1 << 64) - 1) for p in parts)


def sharded_search(search_range: Callable[[int, int], Tuple[int, int, bool]], total: int,
                   group=None) -> Tuple[int, int, bool]:
    """Search [0, total) split over the ranks of `group`.

    ``search_range(first, count) -> (index, makespan, feasible)`` searches one
    contiguous range on this rank (``bf.search_range`` on a GPU).  Returns the
    global (index, makespan, feasible) on every rank.
    """
    import torch.distributed as dist
    rank, world = dist.get_rank(group), dist.get_world_size(group)
    first, count = shard_range(total, rank, world)
    index, makespan, feasible = search_range(first, count) if count else (first, INFEASIBLE, False)
    return unpack_key(min_key_over_ranks(pack_key(index, makespan, feasible), group))


def max_over_ranks(value: float, group=None) -> float:
    """Largest `value` over the ranks (for step times)."""
    import torch
    import torch.distributed as dist
    device = "cuda" if dist.get_backend(group) == "nccl" else "cpu"
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX, group=group)
    return float(t.item())


def gpu_search_range(handle, stream=None) -> Callable[[int, int], Tuple[int, int, bool]]:
    """A ``search_range`` callable over a ``bf`` scenario handle on this rank's GPU."""
    from . import bf

    def run(first: int, count: int) -> Tuple[int, int, bool]:
        r = bf.search_range(handle, first, count, stream)
        return r.index, r.makespan_us, r.feasible
    return run


def sharded_batch(search_batch: Callable[[Sequence], List[Tuple[int, int, bool]]], scenarios: Sequence,
                  group=None) -> List[Tuple[int, int, bool]]:
    """Search every scenario of `scenarios`, split over the ranks of `group`.

    ``search_batch(block) -> [(index, makespan, feasible), ...]`` searches one
    contiguous block of scenarios on this rank (``bf.search_batch`` on a GPU).
    Returns the results of all scenarios, in order, on every rank.
    """
    import torch.distributed as dist
    rank, world = dist.get_rank(group), dist.get_world_size(group)
    first, count = shard_range(len(scenarios), rank, world)
    mine = list(search_batch(scenarios[first:first + count])) if count else []
    parts = [None] * world
    dist.all_gather_object(parts, mine, group=group)
    return [r for part in parts for r in part]


def gpu_search_batch(stream=None) -> Callable[[Sequence], List[Tuple[int, int, bool]]]:
    """A ``search_batch`` callable on this rank's GPU."""
    from . import bf

    def run(block: Sequence) -> List[Tuple[int, int, bool]]:
        return [(r.index, r.makespan_us, r.feasible) for r in bf.search_batch(block, stream)]
    return run
