"""The multi-GPU path's host logic on CPU: two gloo ranks (world size 2).

Replays shard with no data-path collective (each rank replays its own trace
seeds); the job's time is the maximum over ranks and its rate counts every
rank's units.  A record-sharded ranking exchanges each rank's fixed-size
candidate buffer in one all-gather.  These tests run that logic in real
processes over gloo."""
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


def _cands_worker(rank: int, world: int, port: int, out):
    import numpy as np
    import torch
    import torch.distributed as dist
    from paper_2609_09643_gb300 import binding as B
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        nbytes = B.rank_cands_bytes(1024, 512)
        mine = torch.from_numpy(np.random.default_rng(100 + rank).integers(0, 256, nbytes, dtype=np.uint8))
        got = shard.gather_cands(mine)
        out.put((rank, nbytes, mine.numpy().tobytes(), got.numpy().tobytes()))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_gather_candidate_buffers():
    """Every rank ends with the same merge input: the ranks' buffers back to
    back in rank order, each of the size the library states."""
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_cands_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    (_, nb, b0, g0), (_, _, b1, g1) = res
    assert nb == 64 + 16 * (1024 + 2 * 512)
    assert g0 == g1 == b0 + b1


def test_record_slices_partition_the_set():
    for n, world in ((10, 1), (10, 3), (1 << 22, 4), (7, 7)):
        spans = [shard.record_slice(n, r, world) for r in range(world)]
        assert spans[0][0] == 0 and all(c > 0 for _, c in spans)
        assert all(spans[i][0] + spans[i][1] == spans[i + 1][0] for i in range(world - 1))
        assert spans[-1][0] + spans[-1][1] == n
        assert max(c for _, c in spans) - min(c for _, c in spans) <= 1
    with pytest.raises(ValueError):
        shard.record_slice(3, 0, 4)
