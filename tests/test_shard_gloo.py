"""The multi-GPU path's host logic on CPU: two gloo ranks (world size 2).

Replays shard with no data-path collective (each rank replays its own trace
seeds); the job's time is the maximum over ranks and its rate counts every
rank's units.  These tests run that logic in real processes over gloo."""
import os
import socket

import pytest
import torch.multiprocessing as mp

from paper_2609_09643_gb300 import shard


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank: int, world: int, port: int, out):
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ms = 10.0 + 3.5 * rank          # rank 1 is the slowest
        units = 1000 * (rank + 1)       # ranks may process different amounts
        ms_max = shard.max_over_ranks(ms)
        all_units = shard.units_over_ranks(units)
        out.put((rank, ms_max, all_units, shard.job_rate(all_units, 4, ms_max), shard.rank_seeds(rank)))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_reduce_time_and_units():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, ms_max, all_units, rate, seeds in res:
        assert ms_max == 13.5                     # max over ranks, seen by every rank
        assert all_units == [1000, 2000]          # rank order
        assert rate == pytest.approx(3000 * 4 / 13.5e-3)
    s0, s1 = res[0][4], res[1][4]
    assert s0 == list(range(8)) and not set(s0) & set(s1)


def test_single_process_is_identity():
    assert shard.max_over_ranks(7.25) == 7.25
    assert shard.units_over_ranks(42) == [42]
    assert shard.job_rate([10, 20], 2, 1000.0) == 60.0
    with pytest.raises(ValueError):
        shard.job_rate([1], 1, 0.0)
    with pytest.raises(ValueError):
        shard.rank_seeds(-1)
