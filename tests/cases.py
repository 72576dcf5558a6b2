"""Test helpers over the shared workload definitions (synth.workloads): the
oracle jobs that spawned worker processes run."""
from __future__ import annotations

import functools

import synth
from synth.workloads import *  # noqa: F401,F403  (the tests import the workloads from here)
from synth.workloads import large_pool_params, to_oracle


@functools.lru_cache(maxsize=8)
def _coding_trace(seed: int):
    return synth.paper_scale_trace(seed, "coding")


def oracle_sweep_job(job):
    """One oracle replay of the sweep in a worker process: (trace seed,
    params) -> counters.  The worker builds (and keeps) the seed's trace."""
    import oracle
    seed, p = job
    return oracle.replay(_coding_trace(seed), to_oracle(p))


def oracle_rank_job(job):
    """One oracle ranking in a worker process: (record seed, records, params)
    -> victims, moves and moved bytes.  The worker builds the live set."""
    import oracle
    seed, n, p = job
    rec = synth.make_records(seed, n)
    return oracle.rank(rec, p["sigma_q"], p["penalty_q"], p["k"], p["budget_bytes"], p["kv_bytes_per_token"],
                       p["free_fast_tok"], p["free_hbm_tok"], max_moves=max(p["max_moves"], 1))


def oracle_large_pool_job(seed: int):
    """One oracle replay of a large-pool trace in a worker process (the
    worker generates the trace)."""
    import oracle
    return oracle.replay(synth.large_pool_trace(seed), to_oracle(large_pool_params()))
