"""Multi-GPU host logic of the MoCE forward: batch sharding with no exchange.

Every step of the layer is per example (pooling, gate and mixing all act
within one example, Sec. 3.3), and the packed supports and gate parameters are
small constants, so a batch splits across GPUs with no collective on the data
path. Each rank runs the single-GPU forward on its own shard; the only
communication is host-side coordination for measurement (a barrier and the
slowest rank's time).
"""
from __future__ import annotations

import os
from dataclasses import dataclass


@dataclass(frozen=True)
class RankInfo:
    rank: int
    world: int
    local_rank: int


def rank_info() -> RankInfo:
    """Rank, world size and local rank from the torchrun environment (1 process if unset)."""
    return RankInfo(int(os.environ.get("RANK", "0")), int(os.environ.get("WORLD_SIZE", "1")),
                    int(os.environ.get("LOCAL_RANK", "0")))


def shard_bounds(n_total: int, world: int, rank: int) -> tuple[int, int]:
    """Examples [begin, end) of rank's shard when n_total examples split over world ranks.

    Shards differ in size by at most one example; every example belongs to
    exactly one rank.
    """
    if world < 1 or not 0 <= rank < world or n_total < 0:
        raise ValueError("bad shard request")
    base, extra = divmod(n_total, world)
    begin = rank * base + min(rank, extra)
    return begin, begin + base + (1 if rank < extra else 0)


def shard_seed(seed: int, rank: int) -> int:
    """Seed of a rank's synthetic inputs in weak scaling (each rank draws its own batch)."""
    return seed + 1009 * rank


def max_over_ranks(value: float, device=None) -> float:
    """The largest value over all ranks (the slowest rank's time); identity when alone."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(value)
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(units_per_rank: float, world: int, seconds_slowest: float) -> float:
    """Whole-job throughput: the units all ranks processed over the slowest rank's time."""
    if seconds_slowest <= 0:
        raise ValueError("time must be positive")
    return units_per_rank * world / seconds_slowest
