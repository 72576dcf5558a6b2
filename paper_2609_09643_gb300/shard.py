"""Weak-scaling sharding of the batched replay over ranks, one process per GPU.

Replays are independent: each replays its own session trace through its own
state (Algorithm 1 per replay), so ranks exchange no data.  Rank r replays the
parameter sweep on its own trace seeds; the only collective is the reduction
of the timed region to its maximum over ranks, and the job's rate counts the
units every rank processed in that time.  Host logic only: the data path on
every rank is the CUDA library.
"""
from __future__ import annotations

from typing import List, Sequence

SEEDS_PER_RANK = 8


def rank_seeds(rank: int, per_rank: int = SEEDS_PER_RANK) -> List[int]:
    """Trace seeds of one rank: rank 0 has 0..per_rank-1, and the ranks'
    seed sets are disjoint."""
    if rank < 0 or per_rank <= 0:
        raise ValueError("rank >= 0 and per_rank > 0")
    return [per_rank * rank + i for i in range(per_rank)]


def max_over_ranks(value: float, device: str = "cpu") -> float:
    """Maximum of `value` over the process group (identity without one)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(value)
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def units_over_ranks(units: int, device: str = "cpu") -> List[int]:
    """Every rank's unit count (events per step), in rank order."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return [int(units)]
    t = torch.tensor([int(units)], dtype=torch.int64, device=device)
    out = [torch.zeros_like(t) for _ in range(dist.get_world_size())]
    dist.all_gather(out, t)
    return [int(x.item()) for x in out]


def job_rate(units_per_rank: Sequence[int], steps: int, ms_max: float) -> float:
    """Whole-job throughput: the units all ranks processed in `steps` steps,
    over the slowest rank's time."""
    if ms_max <= 0 or steps <= 0:
        raise ValueError("positive time and steps")
    return float(sum(units_per_rank)) * steps / (ms_max / 1e3)
