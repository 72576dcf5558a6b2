"""Resumable replay sweeps.

A sweep is a list of jobs (trace name, replay parameters).  Results are
appended to a JSON-lines file, one row per finished replay, keyed by the
trace name and the canonical form of the parameters; a rerun with the same
file replays only the jobs whose rows are missing.  Rows are written and
flushed a batch at a time, so an interrupted sweep loses at most the batch
in flight; a torn last line (a crash mid-write) is ignored when reading.
"""
from __future__ import annotations

import json
import os
from typing import Callable, Dict, Iterable, List, Sequence, Tuple

Job = Tuple[str, dict]


def job_key(trace_name: str, params: dict) -> str:
    """The row key of a job: its trace name and parameters, canonical JSON."""
    return json.dumps({"trace": trace_name, "params": params}, sort_keys=True, separators=(",", ":"))


def load_rows(path: str) -> Dict[str, dict]:
    """Finished rows of a sweep file by key (missing file: none)."""
    rows: Dict[str, dict] = {}
    if not os.path.exists(path):
        return rows
    with open(path) as f:
        for line in f:
            try:
                row = json.loads(line)
            except json.JSONDecodeError:
                continue  # a torn line from an interrupted write
            if isinstance(row, dict) and "key" in row and "result" in row:
                rows[row["key"]] = row
    return rows


def run_sweep(jobs: Sequence[Job], path: str, runner: Callable[[List[Job]], List[dict]],
              batch: int = 1024) -> List[dict]:
    """Run the jobs not yet in `path` in batches of `batch` through
    runner(jobs) -> results (one dict per job, in order), appending each
    batch's rows; returns the result of every job, in the order given."""
    if batch < 1:
        raise ValueError("batch must be >= 1")
    done = load_rows(path)
    keys = [job_key(t, p) for t, p in jobs]
    todo = [i for i, k in enumerate(keys) if k not in done]
    todo = list(dict.fromkeys(keys[i] for i in todo))  # one run per distinct job
    first = {k: i for i, k in reversed(list(enumerate(keys)))}
    with open(path, "a") as f:
        for b in range(0, len(todo), batch):
            chunk = todo[b:b + batch]
            results = runner([jobs[first[k]] for k in chunk])
            if len(results) != len(chunk):
                raise RuntimeError("runner returned %d results for %d jobs" % (len(results), len(chunk)))
            for k, r in zip(chunk, results):
                t, p = jobs[first[k]]
                row = {"key": k, "trace": t, "params": p, "result": r}
                f.write(json.dumps(row, sort_keys=True) + "\n")
                done[k] = row
            f.flush()
            os.fsync(f.fileno())
    return [done[k]["result"] for k in keys]


def replay_runner(traces: Dict[str, object], stream=None) -> Callable[[List[Job]], List[dict]]:
    """A runner over uploaded binding.Trace handles by name: one
    unison_replay_batch call per batch."""
    from . import binding

    names = list(traces)
    index = {n: i for i, n in enumerate(names)}
    handles = [traces[n] for n in names]

    def run(chunk: List[Job]) -> List[dict]:
        params = [dict(p, trace_idx=index[t]) for t, p in chunk]
        res, _ = binding.replay_batch(handles, params, stream=stream)
        return res

    return run
