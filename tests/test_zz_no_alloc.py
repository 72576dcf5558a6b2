"""The no-allocation replay entry point (unison_replay_batch_noalloc).

It serves callers that cannot allocate device memory (a runtime whose memory
manager owns the whole device budget, or a control loop that cannot pay for
an allocator call).  Its results must equal the ordinary entry point's, call
after call, even though every call reuses one fixed device array.  This file
is collected last so that a failure here leaves every other test already run.
"""
import os
import subprocess
import sys

import pytest

import oracle
import synth
from cases import GIB, MIB, base, to_lib, to_oracle

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def B():
    from paper_2609_09643_gb300 import native
    native.build()
    from paper_2609_09643_gb300 import binding
    return binding


def _workload():
    """Two traces, all six policies, two capacity settings: key streams, TTFT
    values and resident lists all land in the fixed scratch."""
    trs = [synth.tiny_trace(0), synth.paper_scale_trace(3, "general")]
    reps = []
    for ti, (cs, ch, kvb) in enumerate([(512 * MIB, 8 * GIB, 28672), (2 * GIB, 32 * GIB, 131072)]):
        for pol in ("lru", "timeout", "spear", "spear_tide", "belady", "lru_tide"):
            reps.append((ti, base(pol, cs, ch, kvb)))
        # the launch variants: online table, stale snapshot, a signal left out
        reps.append((ti, base("spear_tide", cs, ch, kvb, online=True)))
        reps.append((ti, base("spear", cs, ch, kvb, stale="arrivals", stale_m=4)))
        reps.append((ti, base("spear_tide", cs, ch, kvb, no_hazard=True, stale="gap_start")))
    return trs, reps


def test_noalloc_matches_allocating_entry_point_twice(B):
    import torch
    trs, reps = _workload()
    handles = [B.Trace(t).upload() for t in trs]
    params = [to_lib(p, ti) for ti, p in reps]
    ref, ref_log = B.replay_batch(handles, params, log_capacity=4096)
    n = len(params)
    out = torch.zeros(B.result_nbytes(n), dtype=torch.uint8, device="cuda")
    log = torch.zeros((n, 4096, 2), dtype=torch.int32, device="cuda")
    for call in range(2):
        out.fill_(0xAB)
        log.zero_()
        B.replay_batch_noalloc(handles, params, out, log=log, log_capacity=4096)
        torch.cuda.synchronize()
        got = B.results_from_tensor(out)
        assert got == ref, f"call {call}"
        for i in range(n):
            k = min(ref[i]["log_len"], 4096)
            assert torch.equal(log[i, :k], ref_log[i, :k]), (call, i)
    # and both equal the oracle on every counter, the TTFT statistics and the
    # decision hash, variants included (the oracle keeps a log of the same
    # capacity, so a full log shows in both statuses)
    for i, (ti, p) in enumerate(reps):
        o = oracle.replay(trs[ti], to_oracle(p), log=True, log_capacity=4096)
        for f in ("req_warm", "cold", "hit_s", "hit_h", "miss", "bypass", "evict", "demote", "promote",
                  "tide_demote", "dma_bytes", "tide_calls", "promoted_then_hit_s", "ttft_sum", "ttft_p50_ns",
                  "decision_hash", "vict_n", "vict_diff", "prom_n", "prom_diff", "status"):
            assert got[i][f] == o[f], (i, p["policy"], f, got[i][f], o[f])


def test_noalloc_rejects_batches_beyond_its_scratch(B):
    import torch
    trs = [synth.paper_scale_trace(s, "coding") for s in range(2)]
    handles = [B.Trace(t).upload() for t in trs]
    # 256 replays x 33,596 requests x 8 B of TTFT values alone exceed 32 MiB
    params = [to_lib(base("spear_tide", 2 * GIB, 32 * GIB, 131072), i % 2) for i in range(256)]
    out = torch.zeros(B.result_nbytes(len(params)), dtype=torch.uint8, device="cuda")
    with pytest.raises(B.UnisonError) as e:
        B.replay_batch_noalloc(handles, params, out)
    assert e.value.code == B.ERR_RANGE
    # a batch that fits still runs after the rejection
    ok = params[:8]
    out8 = torch.zeros(B.result_nbytes(8), dtype=torch.uint8, device="cuda")
    B.replay_batch_noalloc(handles, ok, out8)
    torch.cuda.synchronize()
    ref, _ = B.replay_batch(handles, ok)
    assert B.results_from_tensor(out8) == ref


_FRESH = r"""
import sys
sys.path[:0] = [ROOT, ROOT + "/tests"]
import torch
import synth
from cases import GIB, MIB, base, to_lib
from paper_2609_09643_gb300 import binding as B
tr = synth.tiny_trace(0)
h = [B.Trace(tr).upload()]
torch.cuda.synchronize()
params = [to_lib(base(pol, 512 * MIB, 8 * GIB, 28672)) for pol in ("lru", "spear_tide", "belady")]
params.append(to_lib(base("spear_tide", 512 * MIB, 8 * GIB, 28672, online=True)))
out = torch.zeros(B.result_nbytes(len(params)), dtype=torch.uint8, device="cuda")
for call in range(2):
    B.replay_batch_noalloc(h, params, out)  # the first library call of this process on the device
    torch.cuda.synchronize()
    got = B.results_from_tensor(out)
    ref, _ = B.replay_batch(h, params)
    assert got == ref, call
print("fresh-process no-allocation calls match")
"""


def test_noalloc_first_call_in_a_fresh_process(B):
    """The entry point's first call in a process (after only a trace upload)
    sets up the array's address and the side streams itself and still gives
    the allocating entry point's results."""
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    r = subprocess.run([sys.executable, "-c", "ROOT = %r\n" % root + _FRESH], capture_output=True, text=True,
                       timeout=600)
    assert r.returncode == 0, r.stdout + r.stderr
    assert "match" in r.stdout
