"""GPU parity of the batched replay against the CPU oracle.

Bar: bit-exact on every decision (the full decision log where it is
recorded, the decision hash otherwise) and on every counter, including the
TTFT sum and median (integers here, so exact rather than 1e-6)."""
import numpy as np
import pytest

import oracle
import synth
from cases import GIB, MIB, base, to_lib, to_oracle, tiny_case, paper_scale_case, sweep_case, large_pool_params

pytestmark = pytest.mark.gpu

FIELDS = ["events", "req_warm", "cold", "hit_s", "hit_h", "miss", "bypass", "place_s", "place_h", "evict",
          "demote", "promote", "tide_demote", "expire", "tok_hit_s", "tok_hit_h", "tok_miss", "tok_computed",
          "tok_needed", "dma_bytes", "tide_calls", "promoted_then_hit_s", "ttft_sum", "ttft_p50_ns", "ttft_n",
          "decision_hash", "log_len", "vict_n", "vict_diff", "prom_n", "prom_diff", "status"]


@pytest.fixture(scope="module")
def B():
    from paper_2609_09643_gb300 import native
    native.build()
    from paper_2609_09643_gb300 import binding
    return binding


def run_gpu(B, traces, reps, log_capacity=0):
    handles = [B.Trace(t).upload() for t in traces]
    res, log = B.replay_batch(handles, [to_lib(p, ti) for ti, p in reps], log_capacity=log_capacity)
    return res, log, handles


def assert_same(g, o, what=""):
    for f in FIELDS:
        assert g[f] == o[f], (what, f, g[f], o[f])


def assert_same_log(B, log_row, g, o, what=""):
    n = min(g["log_len"], log_row.shape[0])
    ge, gk, gs = B.decode_log(log_row, n)
    oe, ok, os_ = o["log"]
    assert n == len(oe), (what, n, len(oe))
    bad = np.nonzero((ge != oe) | (gk != ok) | (gs != os_))[0]
    assert bad.size == 0, (what, int(bad[0]), (ge[bad[0]], gk[bad[0]], gs[bad[0]]), (oe[bad[0]], ok[bad[0]], os_[bad[0]]))


def test_tiny_all_policies_full_logs(B):
    tr, _ = tiny_case()
    pols = ["lru", "timeout", "spear", "spear_tide", "belady", "lru_tide"]
    reps = [(0, base(p, 512 * MIB, 8 * GIB, 28672)) for p in pols]
    cap = 8 * tr.n_events
    res, log, _ = run_gpu(B, [tr], reps, log_capacity=cap)
    for i, (ti, p) in enumerate(reps):
        o = oracle.replay(tr, to_oracle(p), log=True, log_capacity=cap)
        assert_same(res[i], o, p["policy"])
        assert_same_log(B, log[i], res[i], o, p["policy"])


def test_hand_trace_on_device(B):
    from test_oracle_pins import _hand_trace
    tr, log, counts = _hand_trace("replay_hand_spear.txt")
    p = base("spear", 100, 100, 1, t_p=20_000_000)
    res, lg, _ = run_gpu(B, [tr], [(0, p)], log_capacity=64)
    r = res[0]
    got = list(zip(*(map(int, a) for a in B.decode_log(lg[0], r["log_len"]))))
    assert got == log
    for k, v in counts.items():
        assert r[k] == v, k


def test_hand_tide_trace_on_device(B):
    """The hand-worked SPEAR+TIDE replay (phase-1 promotion beside pinned
    sessions, order and budget stops of the pair loop, the DMA-busy window
    and its exact end, prefetch accuracy) decided the same way on the
    device."""
    from test_oracle_pins import _hand_trace
    tr, log, counts = _hand_trace("replay_hand_tide.txt")
    p = base("spear_tide", 100, 1000, 1, t_p=20_000_000, dma=4)
    res, lg, _ = run_gpu(B, [tr], [(0, p)], log_capacity=64)
    r = res[0]
    got = list(zip(*(map(int, a) for a in B.decode_log(lg[0], r["log_len"]))))
    assert got == log
    for k, v in counts.items():
        assert r[k] == v, k
    assert_same(r, oracle.replay(tr, to_oracle(p)), "hand tide")


def test_paper_scale_30_replays(B):
    trs, reps = paper_scale_case()
    cap = 4 * trs[0].n_events
    res, log, _ = run_gpu(B, trs, reps, log_capacity=cap)
    for i, (ti, p) in enumerate(reps):
        o = oracle.replay(trs[ti], to_oracle(p), log=(i % 6 == 0), log_capacity=cap)
        assert_same(res[i], o, (ti, p["policy"], p["kvb"]))
        if i % 6 == 0:
            assert_same_log(B, log[i], res[i], o, (ti, p["policy"], p["kvb"]))


def test_sweep_1024_replays_all(B):
    """The benchmark's launch configuration: one call over all 1,024 replays,
    every replay checked against the oracle (a spawn pool on the host cores;
    spawned workers do not inherit this process's CUDA context)."""
    import multiprocessing as mp
    import os
    from cases import oracle_sweep_job
    trs, reps = sweep_case()
    res, _, _ = run_gpu(B, trs, reps)
    assert len(res) == 1024
    assert all(r["status"] == 0 for r in res)
    with mp.get_context("spawn").Pool(min(os.cpu_count() or 1, 16)) as pool:
        ores = pool.map(oracle_sweep_job, [(ti, p) for ti, p in reps], chunksize=32)
    for i, o in enumerate(ores):
        assert_same(res[i], o, i)


def test_sweep_iid_gaps_subset(B):
    """The sweep's settings on a trace with independent gaps (gap
    persistence 0: every gap's mixture component and value drawn afresh),
    the workload the bench's `sweep_iid_gaps` rate is measured on: one
    seed's 128 replays in one call, every replay against the oracle."""
    trs, reps = sweep_case(n_seeds=1, gap_persist=0.0)
    res, _, _ = run_gpu(B, trs, reps)
    assert len(res) == 128 and all(r["status"] == 0 for r in res)
    for i, (ti, p) in enumerate(reps):
        assert_same(res[i], oracle.replay(trs[ti], to_oracle(p)), i)


def test_hbm_tier_past_register_capacity(B):
    """SPEAR+TIDE replays around the 160 entries (five a lane) the lean launch
    holds its HBM tier in: with a fast tier of at most 32 entries every replay
    of the call takes the register tiers.  On seed 0 the oracle counts at most
    210 and 192 unpinned HBM sessions for the first two configurations, so
    those replays stop at the 161st entry and run again from their start with
    the tier in shared memory; 126 for the third; and 142 on the trace with
    independent gaps (its fifth slot in use).  Every counter and the decision
    hash against the oracle."""
    trs = [synth.paper_scale_trace(s, "coding") for s in (0, 1)] + [synth.paper_scale_trace(0, "coding", gap_persist=0.0)]
    cfgs = [(28_672, 1 * GIB, 64 * GIB), (131_072, 1 * GIB, 256 * GIB), (28_672, 512 * MIB, 32 * GIB)]
    reps = [(ti, base("spear_tide", cs, ch, kvb)) for ti in range(2) for kvb, cs, ch in cfgs]
    reps += [(2, base("spear_tide", cs, 128 * GIB, 131_072)) for cs in (1 * GIB, 4 * GIB)]
    res, _, _ = run_gpu(B, trs, reps)
    for i, (ti, p) in enumerate(reps):
        assert res[i]["status"] == 0
        assert_same(res[i], oracle.replay(trs[ti], to_oracle(p)), (ti, p["kvb"], p["cap_s"], p["cap_h"]))


@pytest.mark.parametrize("seed", [100, 101])
def test_large_pool_replay(B, seed):
    tr = synth.large_pool_trace(seed)
    p = large_pool_params()
    res, _, _ = run_gpu(B, [tr], [(0, p)])
    assert_same(res[0], oracle.replay(tr, to_oracle(p)), seed)


def test_large_pool_16_replays_one_call(B):
    """The large-pool launch as the benchmark table runs it: many replays, each
    on its own 65,536-session trace, in one call (the tier map without pin
    slots, two CTAs per SM); every replay checked against the oracle in a
    spawn pool."""
    import multiprocessing as mp
    import os
    from cases import oracle_large_pool_job
    seeds = list(range(100, 116))
    trs = [synth.large_pool_trace(s) for s in seeds]
    p = large_pool_params()
    res, _, _ = run_gpu(B, trs, [(i, p) for i in range(len(seeds))])
    with mp.get_context("spawn").Pool(min(os.cpu_count() or 1, 16)) as pool:
        ores = pool.map(oracle_large_pool_job, seeds, chunksize=1)
    for i, o in enumerate(ores):
        assert_same(res[i], o, seeds[i])


POLS = ["lru", "timeout", "spear", "spear_tide", "belady", "lru_tide"]


@pytest.mark.parametrize("caps", [(1 << 60, 1 << 60), (0, 0), (0, 16 * GIB), (2 * GIB, 0), (300 * MIB, 2 * GIB)])
def test_capacity_edges(B, caps):
    tr = synth.paper_scale_trace(5)
    reps = [(0, base(p, caps[0], caps[1], 131072, ttl=0xFFFFFFFF if p == "timeout" else 10_000_000)) for p in POLS]
    res, _, _ = run_gpu(B, [tr], reps)
    for i, (_, p) in enumerate(reps):
        assert_same(res[i], oracle.replay(tr, to_oracle(p)), (caps, p["policy"]))


def test_slot_mode_small_traces(B):
    from test_oracle_pins import _random_seqs, _slot_trace
    trs, reps = [], []
    for k, seq in enumerate(_random_seqs(40, 7)):
        tr, _ = _slot_trace(seq)
        trs.append(tr)
        for slots in (1, 2, 3):
            for pol in ("belady", "lru", "spear"):
                reps.append((k, base(pol, 0, 1 << 60, 1, max_sessions=slots)))
    res, _, _ = run_gpu(B, trs, reps)
    for i, (ti, p) in enumerate(reps):
        assert_same(res[i], oracle.replay(trs[ti], to_oracle(p)), (ti, p["policy"], p["max_sessions"]))


@pytest.mark.parametrize("ttl", [0, 1, 2_000_000, 10_000_000, (1 << 31) - 1, 0xFFFFFFFF])
def test_timeout_ttl(B, ttl):
    tr = synth.paper_scale_trace(6)
    p = base("timeout", 2 * GIB, 32 * GIB, 131072, ttl=ttl)
    res, _, _ = run_gpu(B, [tr], [(0, p)])
    assert_same(res[0], oracle.replay(tr, to_oracle(p)), ttl)


@pytest.mark.parametrize("dma", [0, 1, 6400, 64000, (1 << 32) - 1])
def test_tide_dma_rates(B, dma):
    tr = synth.paper_scale_trace(7)
    reps = [(0, base(pol, 2 * GIB, 32 * GIB, 131072, dma=dma)) for pol in ("spear_tide", "lru_tide")]
    res, _, _ = run_gpu(B, [tr], reps)
    for i, (_, p) in enumerate(reps):
        assert_same(res[i], oracle.replay(tr, to_oracle(p)), (dma, p["policy"]))


@pytest.mark.parametrize("bucket", [1, 3, 8, 64])
def test_bimodal_hazard(B, bucket):
    tr = synth.bimodal_trace(7)
    reps = [(0, base(pol, 1 * GIB, 8 * GIB, 131072, bucket=bucket, ema_num=2, ema_den=9))
            for pol in ("spear", "spear_tide")]
    res, _, _ = run_gpu(B, [tr], reps)
    for i, (_, p) in enumerate(reps):
        assert_same(res[i], oracle.replay(tr, to_oracle(p)), (bucket, p["policy"]))


def test_time_wrap(B):
    """Times near 2^32 us wrap the device's 32-bit clock mid-trace."""
    tr = synth.paper_scale_trace(8)
    shift = np.uint64((1 << 32) - int(tr.arrival_us[len(tr.arrival_us) // 3]))
    sh = synth.Trace(tr.turn_off, tr.arrival_us + shift, tr.completion_us + shift, tr.in_tok, tr.out_tok)
    reps = [(0, base(pol, 2 * GIB, 32 * GIB, 131072, ttl=3_000_000)) for pol in POLS]
    res, _, _ = run_gpu(B, [sh], reps)
    for i, (_, p) in enumerate(reps):
        o = oracle.replay(sh, to_oracle(p))
        assert_same(res[i], o, p["policy"])
        assert o["decision_hash"] == oracle.replay(tr, to_oracle(p))["decision_hash"]


def test_global_list_path(B):
    """Resident lists too large for shared memory live in global memory."""
    tr = synth.make_trace(3, np.full(6000, 4), 0.01, synth.GAP_MIX_CODING)
    reps = [(0, base(pol, 1 << 60, 1 << 60, 1024)) for pol in ("spear_tide", "lru")]
    reps.append((0, base("spear_tide", 400 * MIB, 4 * GIB, 1024)))
    res, _, _ = run_gpu(B, [tr], reps)
    for i, (_, p) in enumerate(reps):
        assert_same(res[i], oracle.replay(tr, to_oracle(p)), i)


def test_global_list_path_spear_tide_only(B):
    """A global-memory launch whose replays are all SPEAR+TIDE runs the
    kernel specialised for that policy."""
    tr = synth.make_trace(3, np.full(6000, 4), 0.01, synth.GAP_MIX_CODING)
    reps = [(0, base("spear_tide", cs, ch, 1024)) for cs, ch in ((1 << 60, 1 << 60), (400 * MIB, 4 * GIB))]
    res, _, _ = run_gpu(B, [tr], reps)
    for i, (_, p) in enumerate(reps):
        assert_same(res[i], oracle.replay(tr, to_oracle(p)), i)


def test_all_six_launch_groups_in_one_call(B):
    """One call with a replay in every launch group (SPEAR+TIDE and other
    policies with lists in shared and in global memory, online table, stale
    snapshot): the groups run concurrently on forked streams, and each replay
    must still equal the oracle, with full decision logs."""
    big = synth.make_trace(3, np.full(6000, 4), 0.01, synth.GAP_MIX_CODING)
    small = synth.paper_scale_trace(2, "general")
    reps = [(0, base("spear_tide", 1 << 60, 1 << 60, 1024)),            # global, SPEAR+TIDE
            (0, base("lru", 1 << 60, 1 << 60, 1024)),                   # global, other
            (1, base("spear_tide", 2 * GIB, 32 * GIB, 131072)),         # shared, SPEAR+TIDE
            (1, base("belady", 2 * GIB, 32 * GIB, 131072)),             # shared, other
            (1, base("spear_tide", 2 * GIB, 32 * GIB, 131072, online=True)),
            (1, base("spear", 2 * GIB, 32 * GIB, 131072, stale="arrivals", stale_m=3))]
    cap = 8 * max(big.n_events, small.n_events)
    trs = [big, small]
    res, log, _ = run_gpu(B, trs, reps, log_capacity=cap)
    for i, (ti, p) in enumerate(reps):
        o = oracle.replay(trs[ti], to_oracle(p), log=True)
        assert_same(res[i], o, i)
        assert_same_log(B, log[i], res[i], o, i)
    # the same replays one per call give the same results
    for i, (ti, p) in enumerate(reps):
        one, _, _ = run_gpu(B, [trs[ti]], [(0, p)])
        assert_same(one[0], res[i], i)


def test_mixed_calls_from_two_host_threads(B):
    """Two host threads issue mixed-policy calls (which fork onto the
    library's side streams) on their own streams at the same time; every
    call's results equal those of a call made alone."""
    import threading
    import torch
    tr = synth.paper_scale_trace(6, "coding")
    h = B.Trace(tr).upload()
    reps = [base(pol, 2 * GIB, 32 * GIB, 131072) for pol in ("spear_tide", "lru", "belady", "spear")]
    params = [to_lib(p) for p in reps]
    ref, _ = B.replay_batch([h], params)
    torch.cuda.synchronize()
    got, errs = [[], []], []

    def worker(k):
        try:
            s = torch.cuda.Stream()
            for _ in range(4):
                with torch.cuda.stream(s):  # the buffer is zeroed on s, before the call
                    out = torch.zeros(B.result_nbytes(len(params)), dtype=torch.uint8, device="cuda")
                B.replay_batch_async([h], params, out, stream=s)
                s.synchronize()
                got[k].append(B.results_from_tensor(out))
        except Exception as e:  # reported on the main thread
            errs.append(e)

    ts = [threading.Thread(target=worker, args=(k,)) for k in range(2)]
    for t in ts:
        t.start()
    for t in ts:
        t.join()
    assert not errs, errs
    for k in range(2):
        assert len(got[k]) == 4
        for res in got[k]:
            for i in range(len(params)):
                assert_same(res[i], ref[i], (k, i))


@pytest.mark.parametrize("n_sessions", [20000, 40000, 240000])
def test_many_sessions_paths(B, n_sessions):
    """20,000 sessions: tier map and pin slots in shared memory.  40,000: the
    tier map alone (completions scan the pinned list).  240,000: no map fits
    beside the lists, so residents are found by a warp-wide search of both
    tiers."""
    tr = synth.make_trace(4, np.full(n_sessions, 3 if n_sessions < 100000 else 2), 0.005, synth.GAP_MIX_GENERAL)
    pols = ("spear_tide", "belady", "timeout") if n_sessions < 100000 else ("spear_tide", "lru")
    reps = [(0, base(pol, 2 * GIB, 16 * GIB, 16384)) for pol in pols]
    res, _, _ = run_gpu(B, [tr], reps)
    for i, (_, p) in enumerate(reps):
        assert_same(res[i], oracle.replay(tr, to_oracle(p)), p["policy"])


def test_degenerate_traces(B):
    """One session with one turn; one session with the most turns a session
    may have (65,535, spanning 40 hours of 32-bit wrapping microseconds);
    every policy at tight, unbounded and zero capacities; and a call with no
    replays."""
    trs = [synth.make_trace(21, np.array([1]), 0.01, synth.GAP_MIX_CODING),
           synth.make_trace(22, np.array([65535]), 0.01, synth.GAP_MIX_CODING)]
    reps = [(ti, base(pol, cs, ch, 28672)) for ti in range(2) for cs, ch in
            ((512 * MIB, 8 * GIB), (1 << 60, 1 << 60), (0, 0)) for pol in POLS]
    res, _, handles = run_gpu(B, trs, reps)
    for i, (ti, p) in enumerate(reps):
        assert_same(res[i], oracle.replay(trs[ti], to_oracle(p)), (ti, p["policy"], p["cap_s"]))
    none, _ = B.replay_batch(handles, [])
    assert none == []


def _random_replays(rng, n_traces, n):
    """n replays with every parameter drawn at random within its valid range:
    policy, capacities from zero to unbounded, KV size, DMA rate, TTL, TTFT
    load, EMA weight, hazard bucket, P_Z, slot limit, and the variants (online
    table, stale snapshot, a signal left out) where the policy allows them."""
    reps = []
    for _ in range(n):
        pol = str(rng.choice(POLS))
        kvb = int(rng.choice([1, 1024, 16384, 28672, 131072, 163840, 1 << 24]))
        cap = lambda: int(rng.choice([0, 1, 64 * MIB, 512 * MIB, 2 * GIB, 16 * GIB, 1 << 60]))
        den = int(rng.choice([1, 2, 5, 10, 33, 4095, 4096, 1 << 20]))
        kw = dict(ema_num=int(rng.integers(0, den + 1)), ema_den=den, bucket=int(rng.choice([1, 2, 3, 8, 60])),
                  penalty=int(rng.choice([0, 1, 500_000_000, (1 << 32) - 1])),
                  ttl=int(rng.choice([0, 1, 2_000_000, (1 << 31) - 1, 0xFFFFFFFF])),
                  dma=int(rng.choice([0, 1, 64_000, (1 << 32) - 1])), load=int(rng.choice([1, 4, 1000])),
                  max_sessions=int(rng.choice([0, 0, 0, 1, 3, 40])))
        if pol in ("spear", "spear_tide"):
            v = int(rng.integers(0, 5))
            if v == 1:
                kw["online"] = True
            elif v == 2:
                kw["stale"] = str(rng.choice(["event", "arrivals", "gap_start"]))
                kw["stale_m"] = int(rng.integers(1, 9))
            elif v == 3:
                kw["no_gap"] = True
            elif v == 4:
                kw["no_hazard"] = bool(rng.integers(0, 2))
                kw["no_gap"] = not kw["no_hazard"]
        reps.append((int(rng.integers(0, n_traces)), base(pol, cap(), cap(), kvb, **kw)))
    return reps


@pytest.mark.parametrize("seed", [20261202, 7, 99])
def test_random_parameters_one_call(B, seed):
    """240 replays with random parameters over four small traces of both gap
    mixes, all in one call (every launch group at once): each replay equals
    the oracle in every counter and its decision hash."""
    rng = np.random.default_rng(seed)
    shapes = ((40, synth.GAP_MIX_CODING), (150, synth.GAP_MIX_GENERAL), (400, synth.GAP_MIX_CODING),
              (90, synth.GAP_MIX_GENERAL))
    trs = [synth.make_trace(40 + i, rng.integers(1, 40, size=n), 0.5, mix) for i, (n, mix) in enumerate(shapes)]
    reps = _random_replays(rng, len(trs), 240)
    res, _, _ = run_gpu(B, trs, reps)
    for i, (ti, p) in enumerate(reps):
        assert_same(res[i], oracle.replay(trs[ti], to_oracle(p)), (i, ti, p))


def test_more_key_streams_than_grid_rows(B):
    """65,600 SPEAR replays with distinct P_Z need 65,600 key streams, more
    than one launch's 65,535 grid rows: the streams are built in two
    launches.  The replays past the boundary use another gap-average weight,
    which changes their decisions, so a second launch reading the first
    launch's streams would fail; replays on both sides equal the oracle."""
    tr, _ = tiny_case()
    reps = [(0, base("spear", 512 * MIB, 8 * GIB, 28672, penalty=7000 * i,
                     ema_num=3 if i < 65535 else 1, ema_den=10 if i < 65535 else 1 << 20)) for i in range(65600)]
    res, _, _ = run_gpu(B, [tr], reps)
    assert all(r["status"] == 0 for r in res)
    for i in list(range(0, 65600, 4099)) + [65533, 65534, 65535, 65536, 65599]:
        assert_same(res[i], oracle.replay(tr, to_oracle(reps[i][1])), i)


def test_log_overflow_reported(B):
    tr, _ = tiny_case()
    p = base("spear_tide", 512 * MIB, 8 * GIB, 28672)
    res, _, _ = run_gpu(B, [tr], [(0, p)], log_capacity=10)
    o = oracle.replay(tr, to_oracle(p), log=True, log_capacity=10)
    assert res[0]["status"] == B.ERR_LOG_FULL == o["status"]
    assert_same(res[0], o)


def test_bad_params_rejected(B):
    tr, _ = tiny_case()
    h = [B.Trace(tr).upload()]
    for bad in (dict(kv_bytes_per_token=0), dict(ema_num=11), dict(penalty_q=1 << 32), dict(ttl_us=1 << 31),
                dict(policy=9), dict(trace_idx=3), dict(hazard_bucket=0)):
        q = to_lib(base("spear", 1 * GIB, 8 * GIB, 28672))
        q.update(bad)
        with pytest.raises(B.UnisonError):
            B.replay_batch(h, [q])


def test_results_on_device_async(B):
    import torch
    trs, reps = paper_scale_case()
    handles = [B.Trace(t).upload() for t in trs]
    out = torch.zeros(B.result_nbytes(len(reps)), dtype=torch.uint8, device="cuda")
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        B.replay_batch_async(handles, [to_lib(p, ti) for ti, p in reps], out, stream=s)
    s.synchronize()
    got = B.results_from_tensor(out)
    ref, _ = B.replay_batch(handles, [to_lib(p, ti) for ti, p in reps])
    assert got == ref


def test_hazard_lut_kernel(B):
    import torch
    for tps in (np.full(64, 12), synth.geometric_turns(3, 5000, 23.7, 2, 200), np.array([1, 2, 2, 3])):
        t = torch.tensor(np.asarray(tps, dtype=np.int32), device="cuda")
        for w in (1, 2, 8, 64):
            sig, hq = B.hazard_lut(t, w)
            oh, osig = oracle.hazard_lut(tps, w)
            assert (sig.cpu().numpy().astype(np.uint16) == osig).all()
            assert (hq.cpu().numpy().astype(np.uint16) == oh).all()


# ---- online hazard table (Sec. V-F) ------------------------------------------

ONLINE_POLS = ("spear", "spear_tide")


def test_online_hazard_tiny_full_logs(B):
    tr, _ = tiny_case()
    reps = [(0, base(pol, 512 * MIB, 8 * GIB, 28672, online=True, bucket=b)) for pol in ONLINE_POLS for b in (1, 3)]
    cap = 8 * tr.n_events
    res, log, _ = run_gpu(B, [tr], reps, log_capacity=cap)
    for i, (_, p) in enumerate(reps):
        o = oracle.replay(tr, to_oracle(p), log=True, log_capacity=cap)
        assert_same(res[i], o, (p["policy"], p["bucket"]))
        assert_same_log(B, log[i], res[i], o, (p["policy"], p["bucket"]))


def test_online_hazard_paper_scale_mixed_batch(B):
    """Online and offline replays of the same settings in one call (the
    online ones run as their own launch): both gap mixes x 3 KV sizes x 2
    policies x buckets 1 and 4.  The online table changes decisions."""
    from cases import KVB_PAPER
    trs = [synth.paper_scale_trace(1, "coding"), synth.paper_scale_trace(1, "general")]
    reps = []
    for ti in range(2):
        for kvb in KVB_PAPER:
            for pol in ONLINE_POLS:
                for b in (1, 4):
                    reps.append((ti, base(pol, 4 * GIB, 64 * GIB, kvb, bucket=b, online=True)))
                    reps.append((ti, base(pol, 4 * GIB, 64 * GIB, kvb, bucket=b)))
    cap = 4 * trs[0].n_events
    res, log, _ = run_gpu(B, trs, reps, log_capacity=cap)
    n_differ = 0
    for i, (ti, p) in enumerate(reps):
        o = oracle.replay(trs[ti], to_oracle(p), log=(i % 8 == 0), log_capacity=cap)
        assert_same(res[i], o, (i, ti, p["policy"], p["kvb"], p["online"]))
        if i % 8 == 0:
            assert_same_log(B, log[i], res[i], o, (i, ti, p["policy"], p["kvb"], p["online"]))
        if p["online"]:
            n_differ += res[i]["decision_hash"] != res[i + 1]["decision_hash"]
    assert n_differ >= len(reps) // 4


def test_online_hazard_two_phase_trace(B):
    """The trace whose online and offline tables coincide once wave 1 has
    completed: full logs against the oracle, online and offline."""
    from test_oracle_pins import _two_phase_trace
    tr = _two_phase_trace()
    reps = [(0, base(pol, 6000 * 131072, 20000 * 131072, 131072, dma=2000, online=on, bucket=b))
            for pol in ONLINE_POLS for on in (True, False) for b in (1, 3)]
    cap = 16 * tr.n_events
    res, log, _ = run_gpu(B, [tr], reps, log_capacity=cap)
    for i, (_, p) in enumerate(reps):
        o = oracle.replay(tr, to_oracle(p), log=True, log_capacity=cap)
        assert_same(res[i], o, i)
        assert_same_log(B, log[i], res[i], o, i)
    assert res[0]["decision_hash"] == res[2]["decision_hash"]  # online == offline at bucket 1


def test_online_hazard_rejected_cases(B):
    tr, _ = tiny_case()
    h = [B.Trace(tr).upload()]
    for pol, flags, err in (("lru", 1, B.ERR_ARG), ("belady", 1, B.ERR_ARG), ("lru_tide", 1, B.ERR_ARG),
                            ("spear", 8, B.ERR_ARG), ("spear", 1 << 31, B.ERR_ARG), ("spear", 3, B.ERR_ARG)):
        q = to_lib(base(pol, 1 * GIB, 8 * GIB, 28672))
        q["flags"] = flags
        with pytest.raises(B.UnisonError) as ei:
            B.replay_batch(h, [q])
        assert ei.value.code == err, (pol, flags)
    # more sessions than an online replay keeps in shared memory
    big = synth.make_trace(5, np.full(40000, 2), 0.005, synth.GAP_MIX_GENERAL)
    hb = [B.Trace(big).upload()]
    with pytest.raises(B.UnisonError) as ei:
        B.replay_batch(hb, [to_lib(base("spear", 1 * GIB, 8 * GIB, 16384, online=True))])
    assert ei.value.code == B.ERR_RANGE


def test_online_attainment_from_device_logs(B):
    """Eq. (attainment) from the device's decision logs (online SPEAR+TIDE,
    offline SPEAR+TIDE, LRU on the paper-scale coding trace) equals the
    oracle's from its own logs."""
    tr = synth.paper_scale_trace(1, "coding")
    ps = [base("spear_tide", 4 * GIB, 64 * GIB, 131072, online=True), base("spear_tide", 4 * GIB, 64 * GIB, 131072),
          base("lru", 4 * GIB, 64 * GIB, 131072)]
    cap = 4 * tr.n_events
    res, log, handles = run_gpu(B, [tr], [(0, p) for p in ps], log_capacity=cap)
    logs = [B.decode_log(log[i], res[i]["log_len"]) for i in range(3)]
    ologs = [oracle.replay(tr, to_oracle(p), log=True, log_capacity=cap)["log"] for p in ps]
    for P in (1, 8, 32):
        got = B.attainment(handles[0], logs, P)
        arr = np.array([[g["sessions_seen"], g["warm"], g["hr_online"], g["hr_offline"], g["hr_lru"],
                         g["attainment"]] for g in got])
        np.testing.assert_array_equal(arr, oracle.attainment(tr, ologs, P)[1])


# ---- stale snapshot of a dual design (Sec. IV-B eq. stale) ---------------------

STALE_MODES = (("event", 0), ("arrivals", 3), ("arrivals", 8), ("gap_start", 0))


def test_stale_snapshot_tiny_full_logs(B):
    tr, _ = tiny_case()
    reps = [(0, base(pol, 512 * MIB, 8 * GIB, 28672, stale=sy, stale_m=m)) for pol in ONLINE_POLS
            for sy, m in STALE_MODES]
    cap = 8 * tr.n_events
    res, log, _ = run_gpu(B, [tr], reps, log_capacity=cap)
    for i, (_, p) in enumerate(reps):
        o = oracle.replay(tr, to_oracle(p), log=True, log_capacity=cap)
        assert_same(res[i], o, (p["policy"], p["stale"], p["stale_m"]))
        assert_same_log(B, log[i], res[i], o, (p["policy"], p["stale"], p["stale_m"]))


def test_stale_snapshot_hand_trace_on_device(B):
    from test_oracle_pins import _hand_trace
    tr, lg, counts = _hand_trace("replay_hand_stale.txt")
    p = base("spear", 300, 0, 1, t_p=20_000_000, stale="arrivals", stale_m=100)
    res, log, _ = run_gpu(B, [tr], [(0, p)], log_capacity=64)
    r = res[0]
    assert list(zip(*(map(int, a) for a in B.decode_log(log[0], r["log_len"])))) == lg
    for k, v in counts.items():
        assert r[k] == v, k


def test_stale_snapshot_paper_scale(B):
    """Both gap mixes x 2 KV sizes x SPEAR / SPEAR+TIDE x the sync modes, in
    one call with the live replays; every-event sync decides as the live
    replay."""
    trs = [synth.paper_scale_trace(1, "coding"), synth.paper_scale_trace(1, "general")]
    reps = []
    for ti in range(2):
        for kvb in (131072, 163840):
            for pol in ONLINE_POLS:
                reps.append((ti, base(pol, 4 * GIB, 64 * GIB, kvb)))
                reps += [(ti, base(pol, 4 * GIB, 64 * GIB, kvb, stale=sy, stale_m=m)) for sy, m in STALE_MODES]
    cap = 4 * trs[0].n_events
    res, log, _ = run_gpu(B, trs, reps, log_capacity=cap)
    for i, (ti, p) in enumerate(reps):
        o = oracle.replay(trs[ti], to_oracle(p), log=(i % 5 == 2), log_capacity=cap)
        assert_same(res[i], o, (i, p["policy"], p["kvb"], p["stale"], p["stale_m"]))
        if i % 5 == 2:
            assert_same_log(B, log[i], res[i], o, (i, p["policy"], p["stale"]))
        if p["stale"] == "event":
            assert res[i]["decision_hash"] == res[i - 1]["decision_hash"] and res[i]["vict_diff"] == 0


def test_stale_snapshot_rejected(B):
    tr, _ = tiny_case()
    h = [B.Trace(tr).upload()]
    for pol, sy, m, online in (("lru", 1, 0, False), ("belady", 3, 0, False), ("spear", 2, 0, False),
                               ("spear", 4, 0, False), ("spear_tide", 1, 0, True)):
        q = to_lib(base(pol, 1 * GIB, 8 * GIB, 28672, online=online))
        q.update(stale_sync=sy, stale_m=m)
        with pytest.raises(B.UnisonError) as ei:
            B.replay_batch(h, [q])
        assert ei.value.code == B.ERR_ARG, (pol, sy, m, online)
    # more sessions than a stale-snapshot replay keeps in shared memory
    big = synth.make_trace(5, np.full(40000, 2), 0.005, synth.GAP_MIX_GENERAL)
    hb = [B.Trace(big).upload()]
    with pytest.raises(B.UnisonError) as ei:
        B.replay_batch(hb, [to_lib(base("spear_tide", 1 * GIB, 8 * GIB, 16384, stale="event"))])
    assert ei.value.code == B.ERR_RANGE


def test_stale_snapshot_with_a_signal_left_out(B):
    """The two variants combine: snapshot keys without the hazard signal, and
    without the gap signal, on the paper-scale coding trace."""
    tr = synth.paper_scale_trace(2, "coding")
    reps = [(0, base(pol, 2 * GIB, 16 * GIB, 131072, stale=sy, stale_m=8, no_gap=ng, no_hazard=not ng))
            for pol in ONLINE_POLS for sy in ("arrivals", "gap_start") for ng in (False, True)]
    res, _, _ = run_gpu(B, [tr], reps)
    for i, (_, p) in enumerate(reps):
        assert_same(res[i], oracle.replay(tr, to_oracle(p)), i)


# ---- signal leave-one-out (Sec. V-D) ----------------------------------------------

def test_signal_leave_one_out_paper_scale(B):
    """Both gap mixes x SPEAR / SPEAR+TIDE x {full, no gap, no hazard, neither},
    in one call (each signal set its own key stream)."""
    trs = [synth.paper_scale_trace(1, "coding"), synth.paper_scale_trace(1, "general")]
    reps = [(ti, base(pol, 4 * GIB, 64 * GIB, 131072, no_gap=ng, no_hazard=nh)) for ti in range(2)
            for pol in ONLINE_POLS for ng in (False, True) for nh in (False, True)]
    cap = 4 * trs[0].n_events
    res, log, _ = run_gpu(B, trs, reps, log_capacity=cap)
    for i, (ti, p) in enumerate(reps):
        o = oracle.replay(trs[ti], to_oracle(p), log=(i % 3 == 1), log_capacity=cap)
        assert_same(res[i], o, (i, p["policy"], p["no_gap"], p["no_hazard"]))
        if i % 3 == 1:
            assert_same_log(B, log[i], res[i], o, (i, p["policy"], p["no_gap"], p["no_hazard"]))
    assert len({r["decision_hash"] for r in res}) == len(res)


def test_signal_special_traces_on_device(B):
    """The pins' traces: gaps of 1 us (no gap signal changes nothing) and
    sessions beyond the table horizon (no hazard signal changes nothing)."""
    from test_oracle_pins import _unit_gap_trace
    tu = _unit_gap_trace()
    th = synth.make_trace(13, 52 + np.arange(30) % 5, 0.4, synth.GAP_MIX_CODING)
    reps = []
    for pol in ONLINE_POLS:
        reps += [(0, base(pol, 3000, 20000, 1)), (0, base(pol, 3000, 20000, 1, no_gap=True))]
        reps += [(1, base(pol, 40000 * 131072, 200000 * 131072, 131072)),
                 (1, base(pol, 40000 * 131072, 200000 * 131072, 131072, no_hazard=True))]
    res, _, _ = run_gpu(B, [tu, th], reps)
    for i, (ti, p) in enumerate(reps):
        assert_same(res[i], oracle.replay([tu, th][ti], to_oracle(p)), i)
        if i % 2:
            assert res[i]["decision_hash"] == res[i - 1]["decision_hash"], i


def test_signal_flags_rejected(B):
    tr, _ = tiny_case()
    h = [B.Trace(tr).upload()]
    for pol, flags in (("lru", 2), ("belady", 4), ("lru_tide", 6), ("spear", 3), ("spear", 8)):
        q = to_lib(base(pol, 1 * GIB, 8 * GIB, 28672))
        q["flags"] = flags
        with pytest.raises(B.UnisonError) as ei:
            B.replay_batch(h, [q])
        assert ei.value.code == B.ERR_ARG, (pol, flags)


# ---- library self-check and host-side fault injection -------------------------------

def test_selftest_division(B):
    """Every divisor 2..4095 at every x < 2^20 and at quotient boundaries up
    to 2^43: the multiply-high division equals the quotient's definition."""
    assert B.selftest_division() == 0


def test_allocation_faults_return_oom(B):
    """A failing device allocation (injected on the host) makes each call
    return UNISON_ERR_OOM and leaves the library usable."""
    import torch
    tr, _ = tiny_case()
    h = [B.Trace(tr).upload()]
    params = [to_lib(base("spear_tide", 512 * MIB, 8 * GIB, 28672))]
    ref, _ = B.replay_batch(h, params)
    B.debug_fail_allocations(1)
    with pytest.raises(B.UnisonError) as ei:
        B.replay_batch(h, params)
    assert ei.value.code == B.ERR_OOM
    assert B.replay_batch(h, params)[0] == ref
    # a trace's first upload
    B.debug_fail_allocations(1)
    t2 = B.Trace(tr)
    with pytest.raises(B.UnisonError) as ei:
        t2.upload()
    assert ei.value.code == B.ERR_OOM
    assert B.replay_batch([t2.upload()], params)[0] == ref
    # the ranking scratch, when a new stream needs its own
    _, sigma = oracle.hazard_lut(synth.geometric_turns(1, 1415, 23.7, 2, 200))
    rec = synth.make_records(3, 5000)
    p = dict(sigma_q=sigma, k=64, penalty_q=500_000_000, budget_bytes=4 << 30, kv_bytes_per_token=131072,
             max_moves=64, free_fast_tok=0, free_hbm_tok=1 << 40)
    dev = B.records_to_device(rec)
    out = B.rank_outputs(rec.n, 64, 64)
    s = torch.cuda.Stream()
    B.debug_fail_allocations(1)
    with pytest.raises(B.UnisonError) as ei:
        B.rank_batch([dev], [p], [out], stream=s)
    assert ei.value.code == B.ERR_OOM
    B.rank_batch([dev], [p], [out], stream=s)
    s.synchronize()
    assert B.rank_result(out)["status"] == 0
    B.debug_fail_allocations(0)


def test_sweep_resume_on_device(B, tmp_path):
    """A sweep interrupted after some rows and rerun equals one run straight
    through, and its rows equal the oracle's results."""
    from paper_2609_09643_gb300 import sweep
    trs = {"tiny0": synth.tiny_trace(0), "tiny1": synth.tiny_trace(1)}
    handles = {k: B.Trace(v).upload() for k, v in trs.items()}
    ps = {pol: base(pol, 512 * MIB, 8 * GIB, 28672) for pol in ("lru", "spear", "spear_tide", "belady")}
    jobs = [(k, to_lib(p)) for k in trs for p in ps.values()]
    full = sweep.run_sweep(jobs, str(tmp_path / "full.jsonl"), sweep.replay_runner(handles), batch=8)
    path = str(tmp_path / "rows.jsonl")
    sweep.run_sweep(jobs[:3], path, sweep.replay_runner(handles), batch=2)
    assert sweep.run_sweep(jobs, path, sweep.replay_runner(handles), batch=2) == full
    for (k, q), r in zip(jobs, full):
        pol = next(p for p in ps.values() if to_lib(p) == q)
        assert r["decision_hash"] == oracle.replay(trs[k], to_oracle(pol))["decision_hash"]
