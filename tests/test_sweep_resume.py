"""Resumable sweeps (checkpoint/resume of result rows), host logic on CPU."""
import json

import pytest

from paper_2609_09643_gb300 import sweep


def _fake(calls):
    def run(chunk):
        calls.append([p["x"] for _, p in chunk])
        return [{"y": p["x"] * p["x"], "t": t} for t, p in chunk]
    return run


def test_rerun_skips_finished_rows(tmp_path):
    path = str(tmp_path / "rows.jsonl")
    jobs = [("a" if i % 2 else "b", {"x": i}) for i in range(10)]
    calls = []
    out = sweep.run_sweep(jobs, path, _fake(calls), batch=4)
    assert out == [{"y": p["x"] ** 2, "t": t} for t, p in jobs]
    assert calls == [[0, 1, 2, 3], [4, 5, 6, 7], [8, 9]]
    calls.clear()
    assert sweep.run_sweep(jobs, path, _fake(calls), batch=4) == out
    assert calls == []
    more = jobs + [("a", {"x": 10})]
    assert sweep.run_sweep(more, path, _fake(calls), batch=4)[-1] == {"y": 100, "t": "a"}
    assert calls == [[10]]


def test_interrupted_sweep_resumes(tmp_path):
    path = str(tmp_path / "rows.jsonl")
    jobs = [("t", {"x": i}) for i in range(9)]
    calls = []

    def failing(chunk):
        if len(calls) == 2:
            raise KeyboardInterrupt
        return _fake(calls)(chunk)

    with pytest.raises(KeyboardInterrupt):
        sweep.run_sweep(jobs, path, failing, batch=3)
    assert len(sweep.load_rows(path)) == 6
    calls.clear()
    out = sweep.run_sweep(jobs, path, _fake(calls), batch=3)
    assert calls == [[6, 7, 8]] and out == [{"y": i * i, "t": "t"} for i in range(9)]


def test_torn_line_and_duplicates(tmp_path):
    path = str(tmp_path / "rows.jsonl")
    jobs = [("t", {"x": 1}), ("t", {"x": 2}), ("t", {"x": 1})]
    calls = []
    sweep.run_sweep(jobs[:1], path, _fake(calls))
    with open(path, "a") as f:
        f.write('{"key": "torn')  # a crash in the middle of a row
    calls.clear()
    out = sweep.run_sweep(jobs, path, _fake(calls))
    assert calls == [[2]]  # x=1 is done, x=2 runs once, the duplicate reuses it
    assert out == [{"y": 1, "t": "t"}, {"y": 4, "t": "t"}, {"y": 1, "t": "t"}]
    with pytest.raises(ValueError):
        sweep.run_sweep(jobs, path, _fake(calls), batch=0)


def test_key_is_canonical():
    assert sweep.job_key("t", {"b": 1, "a": 2}) == sweep.job_key("t", {"a": 2, "b": 1})
    assert sweep.job_key("t", {"a": 1}) != sweep.job_key("u", {"a": 1})
    assert json.loads(sweep.job_key("t", {"a": 1})) == {"trace": "t", "params": {"a": 1}}
