"""Sharding over ranks, one process per GPU.

Replays: weak scaling.  Replays are independent: each replays its own session
trace through its own state (Algorithm 1 per replay), so ranks exchange no
data.  Rank r replays the parameter sweep on its own trace seeds; the only
collective is the reduction of the timed region to its maximum over ranks,
and the job's rate counts the units every rank processed in that time.

One live set ranked by records (Sec. IV-D's scan split over GPUs): rank r
holds the slice record_slice(n, r, world) of the set, ranks it into its
fixed-size candidate buffer (unison_rank_shard), one all-gather brings every
rank's buffer to every rank, and each rank merges them (unison_rank_merge)
into the outputs a single-GPU unison_rank gives for the whole set.

Host logic only: the data path on every rank is the CUDA library.
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


def record_slice(n: int, rank: int, world: int) -> tuple:
    """(index offset, record count) of rank's slice of an n-record set: the
    records split into world contiguous slices, sizes differing by at most
    one, every slice non-empty (n >= world)."""
    if world <= 0 or not 0 <= rank < world or n < world:
        raise ValueError("0 <= rank < world <= n")
    base, extra = divmod(n, world)
    off = rank * base + min(rank, extra)
    return off, base + (1 if rank < extra else 0)


def gather_cands(cands, group=None):
    """All-gather one fixed-size uint8 candidate buffer per rank into a
    buffer of world x its size, in rank order (the merge's input).  Without a
    process group (one GPU) it is the buffer itself."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size(group) == 1:
        return cands
    world = dist.get_world_size(group)
    parts = [torch.empty_like(cands) for _ in range(world)]
    dist.all_gather(parts, cands.contiguous(), group=group)
    return torch.cat(parts)


def rank_sharded(B, rec_slice: dict, n_total: int, params: dict, out: dict, stream=None, group=None) -> None:
    """The whole set's ranking from this rank's slice: shard, all-gather,
    merge (B: the binding module).  Every rank passes the same params and
    gets the same outputs."""
    import torch.distributed as dist
    have = dist.is_available() and dist.is_initialized()
    rank = dist.get_rank(group) if have else 0
    world = dist.get_world_size(group) if have else 1
    off, n = record_slice(n_total, rank, world)
    if int(rec_slice["gap_q"].numel()) != n:
        raise ValueError("the slice does not match this rank's share")
    cands = B.rank_cands(params["k"], params["max_moves"])
    B.rank_shard(rec_slice, off, params, cands, stream)
    gathered = gather_cands(cands, group)
    B.rank_merge(gathered, world, params, out, stream)
