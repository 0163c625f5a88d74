"""Data-parallel sharding of the PHSA hot path across ranks (one GPU each).

Every stage of the path is independent per (sequence, KV head), so ranks
process disjoint sequences and never exchange data. The only collectives are
a barrier and the max-over-ranks of a measured time (``bench.py``).
"""
from __future__ import annotations


def shard_sequences(global_batch: int, world: int, rank: int) -> list[int]:
    """Sequence indices of ``rank``: a contiguous slice, sizes differing by at most 1."""
    if not (0 <= rank < world) or global_batch < 0:
        raise ValueError("bad rank/world/global_batch")
    base, extra = divmod(global_batch, world)
    start = rank * base + min(rank, extra)
    return list(range(start, start + base + (1 if rank < extra else 0)))


def rank_seed(base_seed: int, sequence: int) -> int:
    """Seed of one sequence's synthetic inputs (independent of the rank count)."""
    return base_seed + 7919 * sequence


def max_over_ranks(value: float, device=None) -> float:
    """Maximum of ``value`` over all ranks of the default process group."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(value)
    t = torch.tensor([float(value)], dtype=torch.float64,
                     device=device if device is not None else "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())
