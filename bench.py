#!/usr/bin/env python3
"""Benchmark of the UNISON hot path on GB300.

One step = one batched replay of the parameter sweep (1,024 independent
SPEAR+TIDE replays: 8 trace seeds x 8 tier-capacity pairs x 16 gap-window /
hazard-bucket settings over the paper-scale coding trace, 131,072 B/token)
plus one ranking call over seven 2^24-record live sets (top-1,024 victims and
the TIDE fill at budgets of 1..64 GiB).  Inputs are synthetic (see the synth package) and resident in HBM
before the timed region; an L2 flush (a 256 MiB write) precedes each step.

Prints one JSON line (rank 0).  --impl reference times the CPU oracle on a
bounded sample of the same workload instead.
"""
from __future__ import annotations

import argparse
import csv
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "replay events/s (SPEAR+TIDE batched)"


def rank_traffic(records_per_launch: int):
    """DRAM bytes (read + write) of one rank_kernel launch from the ncu record
    profiles/rank_kernel_traffic.json (one capture, per record), scaled to the
    launch's records; None when rank.cu has changed since the capture (its
    hash no longer matches the recorded one) or the record is missing."""
    import hashlib
    try:
        rec = json.load(open(os.path.join(ROOT, "profiles", "rank_kernel_traffic.json")))
        src = open(os.path.join(ROOT, "paper_2609_09643_gb300", "csrc", "rank.cu"), "rb").read()
        if hashlib.sha256(src).hexdigest()[:16] != rec["rank_cu_sha256_16"]:
            return None
        per = (rec["dram_read_bytes"] + rec["dram_write_bytes"]) / rec["records"]
        return per * records_per_launch
    except (OSError, KeyError, ValueError, ZeroDivisionError):
        return None


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--rank-only", action="store_true", help="time only the ranking leg (profiling)")
    ap.add_argument("--replay-only", action="store_true", help="time only the replay leg (profiling)")
    ap.add_argument("--replays", type=int, default=1024, help="first N replays of the sweep (profiling)")
    ap.add_argument("--rank-n", type=int, default=1 << 24, help="records per live set")
    ap.add_argument("--rank-sets", type=int, default=7, help="live sets per call (<= 7)")
    ap.add_argument("--no-rank-sizes", action="store_true", help="skip the live-set size sweep")
    ap.add_argument("--no-iid", action="store_true", help="skip the sweep on traces with independent gaps")
    ap.add_argument("--online", action="store_true", help="add the online hazard-table report (Sec. V-F)")
    ap.add_argument("--stale", action="store_true", help="add the stale-snapshot (dual design) report")
    ap.add_argument("--ablation", action="store_true", help="add the component/signal/capacity ablations")
    ap.add_argument("--ase", action="store_true", help="add eq. (ase) over the sweep's settings")
    ap.add_argument("--reports", action="store_true", help="all of --online --stale --ablation --ase")
    ap.add_argument("--table", action="store_true",
                    help="per-config table instead of the bench line: GPU events/s, oracle 1-thread and all-core "
                         "events/s, parity, rank GB/s per live-set size")
    ap.add_argument("--table-configs", default="01234", help="which configs the table covers (digits 0-4)")
    return ap.parse_args()


def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


# ---------------------------------------------------------------- clocks ----
CLK_FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")


class ClockSampler:
    def __init__(self, device: int):
        self.path = tempfile.mktemp(suffix=".csv")
        self.proc = None
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(device), f"--query-gpu={CLK_FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=self.f, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.f.close()
        sm, mx, reasons = [], 0.0, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for row in csv.reader(f):
                if len(row) < 9:
                    continue
                try:
                    sm.append(float(row[1]))
                    mx = max(mx, float(row[2]))
                except ValueError:
                    continue
                for n, v in zip(names, row[5:9]):
                    if v.strip().lower() == "active":
                        reasons.add(n)
        os.unlink(self.path)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


# ------------------------------------------------------------- workloads ----
def sweep_workload(rank: int):
    """The 1,024-replay sweep; under torchrun each rank replays it on its own
    trace seeds (rank 0: seeds 0-7, the single-GPU workload)."""
    from synth.workloads import sweep_case, to_lib
    import synth
    from paper_2609_09643_gb300 import shard
    trs, reps = sweep_case()
    if rank:
        trs = [synth.paper_scale_trace(s, "coding") for s in shard.rank_seeds(rank)]
    return trs, reps, [to_lib(p, ti) for ti, p in reps]


RANK_N = 1 << 24  # overridden by --rank-n
RANK_BUDGETS_GIB = (1, 2, 4, 8, 16, 32, 64)
RANK_BYTES_PER_RECORD = 8  # gap average 4 + turn 2 + flags 1 + tier 1: what the filter must read


def rank_workload():
    """Live sets of 2^24 records (the largest live-set size), one per TIDE
    budget 1..64 GiB, each a separate copy in HBM; k = 1,024 victims (every
    k <= 1,024 is a prefix), up to 1,024 moves, no free fast-tier space (pair
    fill only)."""
    import synth
    rec = synth.make_records(4, RANK_N)
    tps = synth.geometric_turns(1, 1415, 23.7, 2, 200)
    return rec, tps


def rank_params(sigma, n_sets=7):
    return [dict(sigma_q=sigma, k=1024, penalty_q=500_000_000, budget_bytes=b << 30, kv_bytes_per_token=131072,
                 max_moves=1024, free_fast_tok=0, free_hbm_tok=1 << 40) for b in RANK_BUDGETS_GIB[:n_sets]]


RANK_SIZES = (1 << 10, 1 << 14, 1 << 18, 1 << 20, 1 << 22, 1 << 24)
RANK_KS = (1, 2, 4, 8, 16, 32, 64, 128, 256, 512, 1024)


def rank_size_sweep(B, host_rec, sigma, stream, peak: float, steps: int = 10, warmup: int = 3):
    """The live-set sizes of the ranking microbenchmark.  At each size one call
    ranks enough distinct sets (slices of the 2^24-record set, at most 64) to
    stream at least 2x the 129 MB L2, so no set is re-read from L2 between
    calls; k cycles through 1..1,024 and the budget through 1..64 GiB.
    call_us = CUDA events around `steps` back-to-back calls on their stream,
    per call (the whole API call: descriptor upload and the kernel); host_us =
    the host's time to issue one call.  frac = GB/s at 8 B/record over the
    measured HBM peak; frac_12B at the plan's 12 B/record."""
    import torch
    out = []
    full = {k: v.to("cuda", non_blocking=True) for k, v in host_rec.items()}
    total = int(full["gap_q"].numel())
    for n in RANK_SIZES:
        n_sets = max(1, min(64, -(-(2 * 129 << 20) // (n * RANK_BYTES_PER_RECORD))))
        sets, params, outs = [], [], []
        for i in range(n_sets):
            off = (i * n) % total if n * n_sets <= total else 0
            if n * n_sets <= total:
                sets.append({k: v[off:off + n] for k, v in full.items()})
            else:  # more records than the 2^24 set holds: separate copies
                sets.append({k: v[:n].clone() for k, v in full.items()})
            k = RANK_KS[i % len(RANK_KS)]
            params.append(dict(sigma_q=sigma, k=k, penalty_q=500_000_000,
                               budget_bytes=RANK_BUDGETS_GIB[i % len(RANK_BUDGETS_GIB)] << 30,
                               kv_bytes_per_token=131072, max_moves=1024, free_fast_tok=0, free_hbm_tok=1 << 40))
            outs.append(B.rank_outputs(n, k, 1024))
        call = B.rank_prepare(sets, params, outs)  # marshalled once: the loop times the device
        for _ in range(warmup):
            call.run(stream)
        torch.cuda.synchronize()
        assert all(B.rank_result(o)["status"] == 0 for o in outs), "rank status"
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        t0 = time.perf_counter()
        for _ in range(steps):
            call.run(stream)
        host_us = 1e6 * (time.perf_counter() - t0) / steps
        e1.record(stream)
        torch.cuda.synchronize()
        call_us = 1e3 * e0.elapsed_time(e1) / steps
        recs = n * n_sets
        gbs = recs * RANK_BYTES_PER_RECORD / (call_us / 1e6) / 1e9
        out.append({"n": n, "sets": n_sets, "call_us": round(call_us, 2), "host_us": round(host_us, 1),
                    "gbs": round(gbs, 1), "frac": round(gbs / peak, 4), "frac_12B": round(1.5 * gbs / peak, 4)})
        del call, sets, outs
    # one set of 2^20 records: the latency of a single call (idle stream)
    n = 1 << 20
    one = [{k: v[:n] for k, v in full.items()}]
    p1 = [dict(sigma_q=sigma, k=1024, penalty_q=500_000_000, budget_bytes=8 << 30, kv_bytes_per_token=131072,
               max_moves=1024, free_fast_tok=0, free_hbm_tok=1 << 40)]
    o1 = [B.rank_outputs(n, 1024, 1024)]
    call = B.rank_prepare(one, p1, o1)
    lat = []
    for i in range(steps + warmup):
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        call.run(stream)
        b.record(stream)
        torch.cuda.synchronize()
        if i >= warmup:
            lat.append(1e3 * a.elapsed_time(b))
    single = {"n": n, "sets": 1, "call_us_median": round(statistics.median(lat), 2)}
    return out, single


def kendall_fp32_vs_fixed(B, host_rec, sigma, stream, n: int = 1 << 20):
    """Kendall tau-b between the fixed-point keys the ranking kernel writes
    (eq. scoreq) and a float32 ranking by the same formula without the
    fixed-point floors, s = g * Lambda / sigma_q + (Lambda - sigma_q) * P_Z /
    Lambda (eq. esp; completed sessions rank first in both), on the first n
    records of the live set.  Reporting only (Sec. IV-C compares the two)."""
    import numpy as np
    import torch
    try:
        from scipy.stats import kendalltau
    except ImportError:
        return None
    part = {k: v[:n].to("cuda") for k, v in host_rec.items()}
    p = dict(sigma_q=sigma, k=1, penalty_q=500_000_000, budget_bytes=0, kv_bytes_per_token=131072, max_moves=0,
             free_fast_tok=0, free_hbm_tok=0)
    out = B.rank_outputs(n, 1, 0, keys=True)
    B.rank_prepare([part], [p], [out]).run(stream)
    torch.cuda.synchronize()
    fixed = out["keys"].cpu().numpy().view(np.uint64)
    g = host_rec["gap_q"][:n].numpy().view(np.uint32).astype(np.float32)
    t = np.minimum(host_rec["turn"][:n].numpy().view(np.uint16), 50)
    sq = np.asarray(sigma, dtype=np.float32)[t]
    lam, pz = np.float32(4095.0), np.float32(500_000_000.0)
    f32 = g * lam / sq + (lam - sq) * pz / lam
    done = (host_rec["flags"][:n].numpy() & 2) != 0
    f32 = np.where(done, np.float32(np.inf), f32).astype(np.float32)
    tau = kendalltau(fixed.astype(np.float64), f32.astype(np.float64))[0]
    return {"tau_b": float(tau), "records": n}


def sweep_ase(B, results, reps, lib_params):
    """Eq. (ase) over the sweep: its 128 settings (fast/HBM capacity pair x
    window x bucket) compared on its 8 traces (seed-major replay order)."""
    n_seeds = 1 + max(ti for ti, _ in reps)
    per = len(reps) // n_seeds
    grid = [[B.stats(results[d * per + c], lib_params[d * per + c]) for d in range(n_seeds)] for c in range(per)]
    vals = B.ase(grid)
    order = sorted(range(per), key=lambda c: -vals[c])
    desc = lambda c: {"cap_fast_gib": lib_params[c]["cap_fast_bytes"] >> 30,
                      "cap_hbm_gib": lib_params[c]["cap_hbm_bytes"] >> 30,
                      "window": lib_params[c]["ema_den"] - 1, "bucket": lib_params[c]["hazard_bucket"]}
    return {"settings": per, "traces": n_seeds, "best": [dict(desc(c), ase=vals[c]) for c in order[:3]],
            "median": sorted(vals)[per // 2], "worst": vals[order[-1]]}


def online_hazard_report(B, stream, steps: int = 3, points: int = 8):
    """Sec. V-F: the paper-scale replays (coding and general gap mixes x 3 KV
    sizes x SPEAR and SPEAR+TIDE, fast 4 GiB / HBM 64 GiB) with a hazard table
    that starts empty and grows at every session completion: device time per
    call, and eq. (attainment) of each against the offline-table and LRU
    replays of the same setting over `points` windows of observed sessions."""
    import math
    import torch
    import synth
    from synth.workloads import GIB, KVB_PAPER, base, to_lib
    mixes = ("coding", "general")
    trs = [synth.paper_scale_trace(1, m) for m in mixes]
    handles = [B.Trace(t).upload(stream) for t in trs]
    settings = [(ti, kvb, pol) for ti in range(2) for kvb in KVB_PAPER for pol in ("spear", "spear_tide")]
    online = [to_lib(base(pol, 4 * GIB, 64 * GIB, kvb, online=True), ti) for ti, kvb, pol in settings]
    offline = [to_lib(base(pol, 4 * GIB, 64 * GIB, kvb), ti) for ti, kvb, pol in settings]
    lru = [to_lib(base("lru", 4 * GIB, 64 * GIB, kvb), ti) for ti, kvb, _ in settings]
    events = sum(2 * trs[ti].n_turns for ti, _, _ in settings)
    out = torch.zeros(B.result_nbytes(len(online)), dtype=torch.uint8, device="cuda")
    for _ in range(2):
        B.replay_batch_async(handles, online, out, stream=stream)
    torch.cuda.synchronize()
    B.profile_enable(True)
    B.profile_read("replay", reset=True)
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(stream)
    for _ in range(steps):
        B.replay_batch_async(handles, online, out, stream=stream)
    b.record(stream)
    torch.cuda.synchronize()
    call_ms = a.elapsed_time(b) / steps
    k_ms, k_n = B.profile_read("replay", reset=True)
    B.profile_enable(False)
    assert all(r["status"] == 0 for r in B.results_from_tensor(out)), "online replay status"

    n = len(settings)
    cap = 4 * max(t.n_events for t in trs)
    res, log = B.replay_batch(handles, online + offline + lru, log_capacity=cap, stream=stream)
    assert all(r["status"] == 0 for r in res), "attainment replay status"
    fin = lambda v: None if v is None or math.isnan(v) else round(v, 4)
    hr = lambda r: (r["hit_s"] + r["hit_h"]) / r["req_warm"] if r["req_warm"] else None
    curves = []
    for i, (ti, kvb, pol) in enumerate(settings):
        logs = [B.decode_log(log[j], res[j]["log_len"]) for j in (i, n + i, 2 * n + i)]
        pts = B.attainment(handles[ti], logs, points)
        curves.append({"trace": mixes[ti], "kv_bytes_per_token": kvb, "policy": pol,
                       "sessions_seen": [p["sessions_seen"] for p in pts],
                       "attainment": [fin(p["attainment"]) for p in pts],
                       "hr_online": fin(hr(res[i])), "hr_offline": fin(hr(res[n + i])), "hr_lru": fin(hr(res[2 * n + i]))})
    return {"replays": n, "events_per_call": events, "call_ms": call_ms,
            "kernel_ms": k_ms / k_n if k_n else None, "events_per_s": events / (call_ms / 1e3),
            "windows": points, "curves": curves}


def stale_snapshot_report(B, stream, steps: int = 3):
    """Sec. IV-B eq. (stale), Tab. org: SPEAR+TIDE on the paper-scale traces
    (coding and general gap mixes x 131,072 and 163,840 B/token, fast 4 GiB /
    HBM 64 GiB) ranked from a register-file copy synced after every event,
    every 8 arrivals, or at every gap_start, against the live ranking: the
    shares of victim and promotion choices that differ, and the shifts of hit
    rate, fast-tier hit share, prefill reduction (points) and AMAT (percent)."""
    import torch
    import synth
    from synth.workloads import GIB, base, to_lib
    mixes = ("coding", "general")
    trs = [synth.paper_scale_trace(1, m) for m in mixes]
    handles = [B.Trace(t).upload(stream) for t in trs]
    modes = (("event", 0), ("arrivals", 8), ("gap_start", 0))
    settings = [(ti, kvb) for ti in range(2) for kvb in (131072, 163840)]
    live = [to_lib(base("spear_tide", 4 * GIB, 64 * GIB, kvb), ti) for ti, kvb in settings]
    stale = [to_lib(base("spear_tide", 4 * GIB, 64 * GIB, kvb, stale=sy, stale_m=m), ti)
             for ti, kvb in settings for sy, m in modes]
    events = sum(2 * trs[ti].n_turns for ti, _ in settings) * len(modes)
    out = torch.zeros(B.result_nbytes(len(stale)), dtype=torch.uint8, device="cuda")
    for _ in range(2):
        B.replay_batch_async(handles, stale, out, stream=stream)
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(stream)
    for _ in range(steps):
        B.replay_batch_async(handles, stale, out, stream=stream)
    b.record(stream)
    torch.cuda.synchronize()
    call_ms = a.elapsed_time(b) / steps
    rs = B.results_from_tensor(out)
    rl, _ = B.replay_batch(handles, live, stream=stream)
    assert all(r["status"] == 0 for r in rs + rl), "stale-snapshot replay status"
    rows = []
    for i, (ti, kvb) in enumerate(settings):
        sl = B.stats(rl[i], live[i])
        hs = lambda r: r["hit_s"] / r["req_warm"] if r["req_warm"] else 0.0
        for j, (sy, m) in enumerate(modes):
            r, q = rs[i * len(modes) + j], stale[i * len(modes) + j]
            st = B.stats(r, q)
            rows.append({"trace": mixes[ti], "kv_bytes_per_token": kvb, "sync": sy if not m else f"every {m} arrivals",
                         "vict_diff_pct": 100.0 * r["vict_diff"] / r["vict_n"] if r["vict_n"] else None,
                         "prom_diff_pct": 100.0 * r["prom_diff"] / r["prom_n"] if r["prom_n"] else None,
                         "d_hr_pp": 100.0 * (st["hit_rate"] - sl["hit_rate"]),
                         "d_fast_pp": 100.0 * (hs(r) - hs(rl[i])),
                         "d_prered_pp": 100.0 * (st["prered"] - sl["prered"]),
                         "d_amat_pct": 100.0 * (st["amat_ps"] / sl["amat_ps"] - 1.0) if sl["amat_ps"] else None,
                         "same_decisions_as_live": r["decision_hash"] == rl[i]["decision_hash"]})
    return {"policy": "spear_tide", "replays": len(stale), "events_per_call": events, "call_ms": call_ms,
            "events_per_s": events / (call_ms / 1e3), "rows": rows}


def ablation_report(B, stream):
    """Sec. V-C..V-E on the paper-scale traces (coding and general mixes,
    131,072 B/token), one batched call for all of it:
    - components (Fig. ablation): LRU, LRU+TIDE, SPEAR, SPEAR+TIDE at fast
      4 GiB / HBM 64 GiB: hit rate, AMAT over LRU's, prefill reduction,
      prefetch accuracy;
    - signals (Fig. signal): SPEAR+TIDE without the gap signal or without the
      hazard signal, shifts of hit rate (points) and AMAT (percent);
    - capacity axes (Tab. robust): SPEAR+TIDE against LRU with HBM swept at
      fast 32K tokens, the fast tier swept at HBM 512K tokens, and the fast
      share of a 256K-token total swept: mean gains over the two traces."""
    import synth
    from synth.workloads import base, to_lib
    kvb, tok = 131072, lambda n: n * 131072
    mixes = ("coding", "general")
    trs = [synth.paper_scale_trace(1, m) for m in mixes]
    handles = [B.Trace(t).upload(stream) for t in trs]
    jobs = []  # (section, label, trace index, params)
    for ti in range(2):
        for pol in ("lru", "lru_tide", "spear", "spear_tide"):
            jobs.append(("component", pol, ti, base(pol, tok(32768), tok(524288), kvb)))
        for lab, ng, nh in (("full", False, False), ("no gap signal", True, False), ("no hazard signal", False, True)):
            jobs.append(("signal", lab, ti, base("spear_tide", tok(32768), tok(524288), kvb, no_gap=ng, no_hazard=nh)))
    axes = [("hbm", f"hbm {h // 1024}K, fast 32K", 32768, h) for h in (131072, 262144, 524288, 1048576)]
    axes += [("fast", f"fast {f // 1024}K, hbm 512K", f, 524288) for f in (8192, 16384, 32768, 65536)]
    axes += [("partition", f"fast share {sh}%", 262144 * sh // 100, 262144 - 262144 * sh // 100)
             for sh in (10, 25, 50, 75)]
    for ax, lab, fs, hb in axes:
        for ti in range(2):
            for pol in ("lru", "spear_tide"):
                jobs.append(("capacity", (ax, lab, pol), ti, base(pol, tok(fs), tok(hb), kvb)))
    params = [to_lib(p, ti) for _, _, ti, p in jobs]
    res, _ = B.replay_batch(handles, params, stream=stream)
    assert all(r["status"] == 0 for r in res), "ablation replay status"
    st = [B.stats(r, q) for r, q in zip(res, params)]
    by = {(j[0], j[1], j[2]): i for i, j in enumerate(jobs)}
    comp = []
    for ti in range(2):
        lru_amat = st[by[("component", "lru", ti)]]["amat_ps"]
        for pol in ("lru", "lru_tide", "spear", "spear_tide"):
            x = st[by[("component", pol, ti)]]
            comp.append({"trace": mixes[ti], "policy": pol, "hit_rate": x["hit_rate"],
                         "amat_over_lru": x["amat_ps"] / lru_amat if lru_amat else None, "prered": x["prered"],
                         "prefetch_acc": x["prefetch_acc"] if pol.endswith("tide") else None})
    sig = []
    for ti in range(2):
        f = st[by[("signal", "full", ti)]]
        for lab in ("no gap signal", "no hazard signal"):
            x = st[by[("signal", lab, ti)]]
            sig.append({"trace": mixes[ti], "variant": lab, "d_hr_pp": 100 * (x["hit_rate"] - f["hit_rate"]),
                        "d_amat_pct": 100 * (x["amat_ps"] / f["amat_ps"] - 1) if f["amat_ps"] else None})
    cap = []
    for ax, lab, fs, hb in axes:
        g_hr, g_amat, g_pre = [], [], []
        for ti in range(2):
            l, u = st[by[("capacity", (ax, lab, "lru"), ti)]], st[by[("capacity", (ax, lab, "spear_tide"), ti)]]
            g_hr.append(100 * (u["hit_rate"] - l["hit_rate"]))
            g_amat.append(100 * (1 - u["amat_ps"] / l["amat_ps"]) if l["amat_ps"] else 0.0)
            g_pre.append(100 * (u["prered"] - l["prered"]))
        cap.append({"axis": ax, "point": lab, "fast_tokens": fs, "hbm_tokens": hb,
                    "mean_hr_gain_pp": sum(g_hr) / 2, "mean_amat_gain_pct": sum(g_amat) / 2,
                    "mean_prered_gain_pp": sum(g_pre) / 2})
    return {"kv_bytes_per_token": kvb, "replays": len(jobs), "components": comp, "signals": sig,
            "capacity_axes": cap, "elapsed_idle_signal": "not built: the hardware scoring contract drops it"}


def cpu_baseline_replay(trs, reps, budget_s: float = 12.0):
    """The oracle as it stands, single-threaded, on a bounded sample of the
    sweep's replays (spread over the batch) until budget_s of CPU work."""
    import oracle
    from synth.workloads import to_oracle
    order = list(range(0, len(reps), 37)) + list(range(1, len(reps), 37))
    ev, n, t0 = 0, 0, time.perf_counter()
    for i in order:
        ti, p = reps[i]
        ev += oracle.replay(trs[ti], to_oracle(p))["events"]
        n += 1
        if time.perf_counter() - t0 > budget_s and n >= 4:
            break
    dt = time.perf_counter() - t0
    return {"value": ev / dt, "unit": "events/s", "cores": 1, "kind": "oracle",
            "sample": f"{n} of the 1,024 sweep replays ({ev} events), single thread, {dt:.1f} s"}


def cpu_baseline_rank(rec, sigma, n: int = 1 << 22):
    """The oracle's ranking (every key, a full sort, the fill) on the first
    2^22 records of one live set, single-threaded."""
    import oracle
    import synth
    sub = synth.Records(*(a[:n].copy() for a in (rec.gap_q, rec.last_ret, rec.turn, rec.kv_tok, rec.tier,
                                                 rec.flags)))
    t0 = time.perf_counter()
    oracle.rank(sub, sigma, 500_000_000, 1024, 64 << 30, 131072, 0, 1 << 40, max_moves=1024)
    dt = time.perf_counter() - t0
    return {"value": n * RANK_BYTES_PER_RECORD / dt / 1e9, "unit": "GB/s", "cores": 1, "kind": "oracle",
            "sample": f"{n} records of one 2^24 live set, k=1024, 64 GiB budget, single thread, {dt:.1f} s"}


def _oracle_replay_job(job):
    """One oracle replay in a worker process (the pool uses spawn)."""
    import oracle
    from synth.workloads import to_oracle
    tr, p = job
    return oracle.replay(tr, to_oracle(p))


def _oracle_rank_job(job):
    import oracle
    import synth
    rec, sigma, n = job
    sub = synth.Records(*(a[:n].copy() for a in (rec.gap_q, rec.last_ret, rec.turn, rec.kv_tok, rec.tier,
                                                 rec.flags)))
    oracle.rank(sub, sigma, 500_000_000, 1024, 64 << 30, 131072, 0, 1 << 40, max_moves=1024)
    return n


def _large_trace_job(seed):
    """One large-pool trace, generated in a worker process."""
    import synth
    return synth.large_pool_trace(seed)


def _oracle_large_job(seed):
    """One large-pool oracle replay in a worker (it generates its own trace)."""
    import oracle
    import synth
    from synth.workloads import large_pool_params, to_oracle
    return oracle.replay(synth.large_pool_trace(seed), to_oracle(large_pool_params()))


def large_pool_table(B, pool, stream, fields, cores):
    """Config 3 at full size: 256 replays (seeds 100-355) in one launch, each
    on its own 65,536-session trace; every replay checked against the oracle.
    Traces are generated in the worker pool and their handles built on host
    threads, so the parent never holds more than the pinned upload copies."""
    from concurrent.futures import ThreadPoolExecutor
    import torch
    from synth.workloads import large_pool_params, to_lib, to_oracle
    import oracle
    import synth
    seeds = list(range(100, 356))
    with ThreadPoolExecutor(cores) as ex:
        futs = [ex.submit(lambda t: B.Trace(t), tr) for tr in pool.imap(_large_trace_job, seeds, chunksize=1)]
        handles = [f.result() for f in futs]
    for h in handles:
        h.upload(stream)
    ev = sum(2 * h.info()[1] for h in handles)
    params = [to_lib(large_pool_params(), i) for i in range(len(seeds))]
    res_dev = torch.zeros(B.result_nbytes(len(params)), dtype=torch.uint8, device="cuda")
    B.replay_batch_async(handles, params, res_dev, stream=stream)
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    steps = 2
    a.record(stream)
    for _ in range(steps):
        B.replay_batch_async(handles, params, res_dev, stream=stream)
    b.record(stream)
    torch.cuda.synchronize()
    gpu = ev * steps / (a.elapsed_time(b) / 1e3)
    res = B.results_from_tensor(res_dev)
    del handles, res_dev
    spent, ev1, n1 = 0.0, 0, 0
    for sd in seeds:
        tr = synth.large_pool_trace(sd)
        t0 = time.perf_counter()
        ev1 += oracle.replay(tr, to_oracle(large_pool_params()))["events"]
        spent += time.perf_counter() - t0
        n1 += 1
        if spent > 10.0:
            break
    one = ev1 / spent
    t0 = time.perf_counter()
    ores = pool.map(_oracle_large_job, seeds, chunksize=1)
    allc = sum(r["events"] for r in ores) / (time.perf_counter() - t0)
    bad = [sd for sd, r, g in zip(seeds, ores, res) if any(g[f] != r[f] for f in fields)]
    return {"config": "3 large pool (256 replays, seeds 100-355)", "replays": len(seeds), "events_per_launch": ev,
            "gpu_events_per_s": gpu, "oracle_1core_events_per_s": one,
            "oracle_1core_sample": f"{n1} replays",
            "oracle_allcore_events_per_s": allc,
            "oracle_allcore_sample": "all 256 (each worker generates its trace inside the timed region)",
            "cores": cores,
            "parity": f"{len(seeds) - len(bad)}/{len(seeds)} replays identical" + (f", differ: {bad[:5]}" if bad else "")}


def config_table(args):
    """Configs 0-3 (replays) and 4 (ranking): device events/s of one batched
    launch (CUDA events, warm), the oracle on one core and on all host cores
    (a spawn pool, one replay per task) over a stated sample, and parity of
    every replay the oracle ran (all counters and the decision hash)."""
    import multiprocessing as mp
    import torch
    import synth
    from synth.workloads import tiny_case, paper_scale_case, sweep_case, large_pool_params, to_lib, to_oracle
    import oracle
    from paper_2609_09643_gb300 import native
    torch.cuda.set_device(0)
    native.build()
    from paper_2609_09643_gb300 import binding as B
    cores = os.cpu_count() or 1
    pool = mp.get_context("spawn").Pool(cores)
    stream = torch.cuda.current_stream()
    tr0, ps0 = tiny_case()
    trs2, reps2 = sweep_case()
    cfgs = [("0 tiny", [tr0], [(0, p) for p in ps0], 50, "all 4"),
            ("1 paper-scale", *paper_scale_case(), 10, "all 30"),
            ("2 sweep", trs2, reps2, 5, "32 replays spread over the 1,024")]
    cfgs = [c for c in cfgs if c[0][0] in args.table_configs]
    fields = ["events", "req_warm", "hit_s", "hit_h", "miss", "evict", "demote", "promote", "tide_demote",
              "tok_computed", "ttft_sum", "ttft_p50_ns", "decision_hash", "status"]
    out = []
    for name, trs, reps, steps, sample in cfgs:
        handles = [B.Trace(t).upload(stream) for t in trs]
        params = [to_lib(p, ti) for ti, p in reps]
        ev = sum(2 * trs[ti].n_turns for ti, _ in reps)
        res_dev = torch.zeros(B.result_nbytes(len(params)), dtype=torch.uint8, device="cuda")
        B.replay_batch_async(handles, params, res_dev, stream=stream)
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(steps):
            B.replay_batch_async(handles, params, res_dev, stream=stream)
        b.record(stream)
        torch.cuda.synchronize()
        gpu = ev * steps / (a.elapsed_time(b) / 1e3)
        res = B.results_from_tensor(res_dev)
        pick = list(range(len(reps))) if not name.startswith("2") else [int(i * 1024 / 32) for i in range(32)]
        # one core: a bounded part of the sample, in this process
        t0, ev1, n1 = time.perf_counter(), 0, 0
        for i in pick:
            ti, p = reps[i]
            ev1 += oracle.replay(trs[ti], to_oracle(p))["events"]
            n1 += 1
            if time.perf_counter() - t0 > 10.0:
                break
        one = ev1 / (time.perf_counter() - t0)
        # all cores: the whole sample
        t0 = time.perf_counter()
        ores = pool.map(_oracle_replay_job, [(trs[reps[i][0]], reps[i][1]) for i in pick], chunksize=1)
        allc = sum(r["events"] for r in ores) / (time.perf_counter() - t0)
        bad = [i for i, r in zip(pick, ores) if any(res[i][f] != r[f] for f in fields)]
        out.append({"config": name, "replays": len(reps), "events_per_launch": ev, "gpu_events_per_s": gpu,
                    "oracle_1core_events_per_s": one, "oracle_1core_sample": f"{n1} replays",
                    "oracle_allcore_events_per_s": allc, "oracle_allcore_sample": sample, "cores": cores,
                    "parity": f"{len(pick) - len(bad)}/{len(pick)} replays identical" + (f", differ: {bad[:5]}" if bad else "")})
        del handles, res_dev
    if "3" in args.table_configs:
        out.append(large_pool_table(B, pool, stream, fields, cores))
    pk = json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json"))).get("hbm_gbs") or 6800.0
    if "4" not in args.table_configs:
        pool.close()
        print(json.dumps({"table": out, "peak_hbm_gbs": pk}), flush=True)
        return
    # config 4: the ranking at each live-set size (device), the oracle on 2^22 records
    rec, tps = rank_workload()
    tps_dev = torch.tensor(tps.astype("int32"), device="cuda")
    sig_dev, _ = B.hazard_lut(tps_dev, 1)
    sigma = sig_dev.cpu().numpy().astype("uint16")
    host_rec = {k: v.pin_memory() for k, v in B.records_to_device(rec, device="cpu").items()}
    sizes, single = rank_size_sweep(B, host_rec, sigma, stream, pk)
    one = cpu_baseline_rank(rec, sigma)
    t0 = time.perf_counter()
    n = sum(pool.map(_oracle_rank_job, [(rec, sigma, 1 << 22)] * cores, chunksize=1))
    allc = n * RANK_BYTES_PER_RECORD / (time.perf_counter() - t0) / 1e9
    pool.close()
    out.append({"config": "4 rank", "gpu": sizes, "gpu_single_set": single,
                "oracle_1core_gbs": one["value"], "oracle_allcore_gbs": allc, "cores": cores,
                "oracle_sample": "2^22 records of one 2^24 live set per core, k=1,024, full sort + fill"})
    print(json.dumps({"table": out, "peak_hbm_gbs": pk}), flush=True)


def run_reference(args):
    world, rank, _ = dist_env()
    if rank != 0:
        return
    import oracle
    from synth.workloads import to_oracle
    trs, reps, _ = sweep_workload(0)
    per_step = 8
    order = list(range(0, len(reps), 127))
    times, evs = [], []
    for step in range(args.warmup + args.steps):
        t0 = time.perf_counter()
        ev = 0
        for j in range(per_step):
            ti, p = reps[order[(step * per_step + j) % len(order)]]
            ev += oracle.replay(trs[ti], to_oracle(p))["events"]
        dt = time.perf_counter() - t0
        if step >= args.warmup:
            times.append(dt)
            evs.append(ev)
    v = sum(evs) / sum(times)
    line = {"impl": "reference", "metric": METRIC, "value": v, "unit": "events/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000 * sum(times) / len(times),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "int64",
            "data": "synthetic",
            "config": {"workload": "sweep-1024 (8 seeds x 8 capacity pairs x 16 window/bucket settings, "
                                   "paper-scale coding trace, gap persistence rho = 0.7, 131072 B/token, "
                                   "SPEAR+TIDE)",
                       "sample_per_step": f"{per_step} replays", "l2": "n/a (CPU)"},
            "cpu_baseline": {"kind": "oracle", "cores": 1, "value": v, "unit": "events/s",
                             "sample": f"{per_step} sweep replays per step, single-threaded C oracle"},
            "e2e": {"value": v, "unit": "events/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def main():
    global RANK_N
    args = parse()
    RANK_N = args.rank_n
    if args.impl == "reference":
        return run_reference(args)
    if args.table:
        return config_table(args)
    import torch
    world, rank, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    else:
        torch.cuda.set_device(0)
    dev = torch.cuda.current_device()
    from paper_2609_09643_gb300 import native
    native.build()
    from paper_2609_09643_gb300 import binding as B

    trs, reps, lib_params = sweep_workload(rank)
    if args.replays < len(reps):  # evenly spread subset, for profiling runs
        pick = [int(i * len(reps) / args.replays) for i in range(args.replays)]
        reps = [reps[i] for i in pick]
        lib_params = [lib_params[i] for i in pick]
    stream = torch.cuda.current_stream()
    handles = [B.Trace(t).upload(stream) for t in trs]
    n_rep = len(lib_params)
    events_per_step = sum(2 * trs[ti].n_turns for ti, _ in reps)
    res_dev = torch.zeros(B.result_nbytes(n_rep), dtype=torch.uint8, device="cuda")
    flush = torch.empty(256 << 20, dtype=torch.uint8, device="cuda")

    # ranking leg: survival table from the paper-scale turn law, on the device
    rec, tps = rank_workload()
    tps_dev = torch.tensor(tps.astype("int32"), device="cuda")
    sig_dev, _ = B.hazard_lut(tps_dev, 1)
    sigma = sig_dev.cpu().numpy().astype("uint16")
    r_params = rank_params(sigma, args.rank_sets)
    host_rec = B.records_to_device(rec, device="cpu")
    host_rec = {k: v.pin_memory() for k, v in host_rec.items()}
    rank_sets = [{k: v.to("cuda", non_blocking=True) for k, v in host_rec.items()} for _ in r_params]
    rank_outs = [B.rank_outputs(RANK_N, p["k"], p["max_moves"]) for p in r_params]
    rank_bytes = len(r_params) * RANK_N * RANK_BYTES_PER_RECORD

    rank_call = B.rank_prepare(rank_sets, r_params, rank_outs) if not args.replay_only else None
    rank_marks = []  # (start, end) events around each timed rank call

    def step(mark=False):
        flush.zero_()
        if not args.rank_only:
            B.replay_batch_async(handles, lib_params, res_dev, stream=stream)
        if not args.replay_only:
            if mark:
                a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                a.record(stream)
            rank_call.run(stream)
            if mark:
                b.record(stream)
                rank_marks.append((a, b))

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    ase = None
    if not args.rank_only:
        res = B.results_from_tensor(res_dev)
        assert all(r["status"] == 0 for r in res), "replay status"
        if len(res) == 1024 and (args.ase or args.reports):
            ase = sweep_ase(B, res, reps, lib_params)
    if not args.replay_only:
        assert all(B.rank_result(o)["status"] == 0 for o in rank_outs), "rank status"

    def barrier():
        if world > 1:
            torch.distributed.barrier()

    barrier()
    torch.cuda.synchronize()
    clk = ClockSampler(dev)
    B.profile_enable(True)
    for kname in ("replay", "key_stream", "ttft_median", "rank"):
        B.profile_read(kname, reset=True)
    launches0 = B.launch_count()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        step(mark=True)
    e1.record(stream)
    torch.cuda.synchronize()
    barrier()
    ms = e0.elapsed_time(e1)
    launches = B.launch_count() - launches0
    rep_ms, rep_n = B.profile_read("replay", reset=True)
    ks_ms, ks_n = B.profile_read("key_stream", reset=True)
    md_ms, md_n = B.profile_read("ttft_median", reset=True)
    rk_ms, rk_n = B.profile_read("rank", reset=True)
    B.profile_enable(False)
    clocks = clk.stop()
    from paper_2609_09643_gb300 import shard
    ms = shard.max_over_ranks(ms, device="cuda")
    units = shard.units_over_ranks(events_per_step, device="cuda")
    value = shard.job_rate(units, args.steps, ms) if not args.rank_only else None
    peaks = {}
    try:
        peaks = json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    except Exception:
        pass
    hbm_peak = peaks.get("hbm_gbs") or 6800.0

    sizes = single = None
    tau = None
    if not args.replay_only:
        tau = kendall_fp32_vs_fixed(B, host_rec, sigma, stream)
    if not args.replay_only and not args.no_rank_sizes:
        sizes, single = rank_size_sweep(B, host_rec, sigma, stream, hbm_peak)

    # the sweep on traces whose gaps are drawn independently (no per-session
    # persistence: every gap's mixture component and value drawn afresh),
    # timed like the main leg
    iid = None
    if not (args.no_iid or args.rank_only or world > 1):
        from synth.workloads import sweep_case, to_lib
        trs0, reps0 = sweep_case(gap_persist=0.0)
        h0 = [B.Trace(t).upload(stream) for t in trs0]
        p0 = [to_lib(p, ti) for ti, p in reps0]
        ev0 = sum(2 * trs0[ti].n_turns for ti, _ in reps0)
        r0 = torch.zeros(B.result_nbytes(len(p0)), dtype=torch.uint8, device="cuda")
        for _ in range(2):
            B.replay_batch_async(h0, p0, r0, stream=stream)
        torch.cuda.synchronize()
        assert all(r["status"] == 0 for r in B.results_from_tensor(r0)), "replay status"
        n_iid = max(3, args.steps // 2)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(n_iid):
            flush.zero_()
            B.replay_batch_async(h0, p0, r0, stream=stream)
        b.record(stream)
        torch.cuda.synchronize()
        iid = {"gap_persistence": 0.0, "events_per_step": ev0, "steps": n_iid,
               "ms_per_step": round(a.elapsed_time(b) / n_iid, 3),
               "events_per_s": ev0 * n_iid / (a.elapsed_time(b) / 1e3)}
        for h in h0:
            h.close()

    rep_all = args.reports
    online = None
    if (args.online or rep_all) and not (args.rank_only or args.replay_only) and rank == 0:
        online = online_hazard_report(B, stream)
    stale = None
    if (args.stale or rep_all) and not (args.rank_only or args.replay_only) and rank == 0:
        stale = stale_snapshot_report(B, stream)
    ablation = None
    if (args.ablation or rep_all) and not (args.rank_only or args.replay_only) and rank == 0:
        ablation = ablation_report(B, stream)

    # end to end through the public API, every step: the step's traces and live
    # sets copied from pinned host memory to the device, the replay sweep and
    # the rank call, and their results copied back and read on the host.  Two
    # input/output buffers let step i+1's copies (on a copy stream) overlap
    # step i's kernels; step i's results are read while step i+1 runs.
    e2e = None
    if not args.no_e2e and not args.rank_only:
        copy_stream = torch.cuda.Stream()
        h2d = sum(h.device_bytes for h in handles) + len(rank_sets) * sum(
            v.numel() * v.element_size() for v in host_rec.values())
        d2h = B.result_nbytes(n_rep) + sum(o["victims"].numel() * 4 + o["promote"].numel() * 4 +
                                           o["demote"].numel() * 4 + o["counts"].numel() * 4 + 8 for o in rank_outs)
        bufs = []
        for bi_ in range(2):
            hb = handles if bi_ == 0 else [B.Trace(t).upload(stream) for t in trs]
            sb = rank_sets if bi_ == 0 else [{k: torch.empty_like(v) for k, v in s0.items()} for s0 in rank_sets]
            ob = rank_outs if bi_ == 0 else [B.rank_outputs(RANK_N, p["k"], p["max_moves"]) for p in r_params]
            out_host = {"res": torch.empty(B.result_nbytes(n_rep), dtype=torch.uint8).pin_memory(),
                        "rank": [{k: torch.empty(v.shape, dtype=v.dtype).pin_memory() for k, v in o.items() if v is not None}
                                 for o in ob]}
            bufs.append(dict(handles=hb, sets=sb, outs=ob, call=B.rank_prepare(sb, r_params, ob),
                             res=torch.zeros(B.result_nbytes(n_rep), dtype=torch.uint8, device="cuda"),
                             host=out_host, ev_in=torch.cuda.Event(), ev_out=torch.cuda.Event(), used=False))
        torch.cuda.synchronize()

        def read(buf):  # the host reads one step's results
            buf["ev_out"].synchronize()
            res = B.results_from_tensor(buf["host"]["res"])
            assert all(r["status"] == 0 for r in res), "replay status"
            assert all(int(h["counts"][3]) == 0 for h in buf["host"]["rank"]), "rank status"

        t0 = time.perf_counter()
        for step_i in range(args.steps):
            buf = bufs[step_i % 2]
            with torch.cuda.stream(copy_stream):
                if buf["used"]:
                    copy_stream.wait_event(buf["ev_out"])  # step i-2 is done with this buffer
                for h in buf["handles"]:
                    h.upload(copy_stream)
                for dst in buf["sets"]:
                    for k, v in host_rec.items():
                        dst[k].copy_(v, non_blocking=True)
                buf["ev_in"].record(copy_stream)
            stream.wait_event(buf["ev_in"])
            B.replay_batch_async(buf["handles"], lib_params, buf["res"], stream=stream)
            buf["call"].run(stream)
            with torch.cuda.stream(stream):
                buf["host"]["res"].copy_(buf["res"], non_blocking=True)
                for ho, o in zip(buf["host"]["rank"], buf["outs"]):
                    for k, hv in ho.items():
                        hv.copy_(o[k], non_blocking=True)
            buf["ev_out"].record(stream)
            if step_i > 0:
                read(bufs[(step_i - 1) % 2])
            buf["used"] = True
        read(bufs[(args.steps - 1) % 2])
        torch.cuda.synchronize()
        dt = time.perf_counter() - t0
        e2e = {"value": shard.job_rate(units, args.steps, 1e3 * shard.max_over_ranks(dt, device="cuda")),
               "unit": "events/s", "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
               "pipelined": "two buffers: step i+1's copies overlap step i's kernels"}
        del bufs

    avg_rep_ms = rep_ms / max(rep_n, 1) if rep_n else float("nan")
    # 16 B event + 4 B previous size + 8 B key + 4 B gap average + 8 B key
    # before each arrival (half the events): 36 B/event
    alg_bytes = events_per_step * 36
    replay_roof = None if not rep_n else {"bound": "latency", "kernel": "replay_kernel", "avg_ms": avg_rep_ms,
                   "ns_per_event_per_replay": 1e6 * avg_rep_ms / (events_per_step / n_rep),
                   "hbm_gbs": alg_bytes / (avg_rep_ms / 1e3) / 1e9, "launches_timed": rep_n,
                   "share_of_step": avg_rep_ms * args.steps / ms if ms else None,
                   "key_stream_avg_ms": ks_ms / max(ks_n, 1), "ttft_median_avg_ms": md_ms / max(md_n, 1)}
    if replay_roof is not None:
        # The launch ends with its slowest replay: its cycles per event, against
        # the chain an event needs with both tiers in the warp's registers and
        # the pin list in shared memory (about 17 dependent steps of about 30
        # cycles each: the event's and its key's loads, the lookup ballot and
        # entry shuffle, the erase shuffle, pin slot, pin entry and its store,
        # a demotion's pop, the HBM search ballot and insert shuffle, TIDE's
        # two heads and its insert's ballot and shuffle).
        mhz = (clocks or {}).get("sm_mhz") or 2070.0
        replay_roof["cycles_per_event_slowest_replay"] = avg_rep_ms * 1e3 * mhz / (events_per_step / n_rep)
        replay_roof["floor_cycles_per_event"] = 17 * 30
        replay_roof["floor_basis"] = ("17 dependent steps per event x ~30 cycles: shared-memory loads (event, key, "
                                      "pin slot and entry) and the register tiers' ballots and shuffles (lookup, "
                                      "erase, demotion, HBM insert, TIDE heads and insert)")
    avg_rk = rk_ms / max(rk_n, 1) if rk_n else float("nan")
    achieved = rank_bytes / (avg_rk / 1e3) / 1e9 if rk_n else float("nan")
    n_rec = len(r_params) * RANK_N
    # the whole ranking call is one kernel: sample, filter and finish of every set
    roofline = {"bound": "hbm", "kernel": "rank_kernel", "achieved": achieved, "peak": hbm_peak,
                "unit": "GB/s", "frac": achieved / hbm_peak,
                "peak_source": "measured (MEASURED_PEAKS.json hbm_gbs, burst copy)" if peaks.get("hbm_gbs")
                else "fallback 6.8 TB/s", "traffic": rank_traffic(n_rec),
                "traffic_source": "profiles/rank_kernel_traffic.json (ncu dram bytes per record, scaled)",
                "avg_ms": avg_rk, "launches_timed": rk_n, "algorithmic_bytes_per_launch": rank_bytes,
                "bytes_per_record": RANK_BYTES_PER_RECORD, "records_per_launch": n_rec,
                "at_12B_per_record": {"achieved": 1.5 * achieved, "frac": 1.5 * achieved / hbm_peak},
                "bytes_reading": "8 B/record streamed (gap 4, turn 2, flags 1, tier 1); sizes are gathered "
                                 "only for the <= 4,096 movable records per list, so kv_tok is not streamed"}
    call_ms = (sum(a.elapsed_time(b) for a, b in rank_marks) / len(rank_marks)) if rank_marks else float("nan")
    rank_leg = {"sets_per_call": len(r_params), "records_per_set": RANK_N, "k": 1024,
                "call_ms": call_ms, "kernel_ms": avg_rk,
                "call_gbs": rank_bytes / (call_ms / 1e3) / 1e9,
                "call_frac_of_peak": rank_bytes / (call_ms / 1e3) / 1e9 / hbm_peak,
                "call_frac_of_peak_12B": 1.5 * rank_bytes / (call_ms / 1e3) / 1e9 / hbm_peak}
    if rank != 0:
        return
    cpu = None if (args.no_cpu_baseline or world > 1) else cpu_baseline_replay(trs, reps)
    # the whole ranking call's fraction per live-set size as flat keys (8 B/record)
    flat = {"rank_call_frac_2p%d_x%d" % (z["n"].bit_length() - 1, z["sets"]): z["frac"]
            for z in sizes or [] if z["n"] >= (1 << 20)}
    line = {"metric": METRIC, "value": value, "unit": "events/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "int64", "data": "synthetic",
            "config": {"workload": "sweep-1024 (8 seeds x 8 capacity pairs x 16 window/bucket settings, "
                                   "paper-scale coding trace, gap persistence rho = 0.7, 131072 B/token, "
                                   "SPEAR+TIDE)",
                       "replays": n_rep, "events_per_step": events_per_step,
                       "l2": "flushed before every step (256 MiB write, inside the timed region)"},
            "rank_call_frac_of_peak": rank_leg["call_frac_of_peak"], **flat,
            "roofline": roofline, "rank": rank_leg, "rank_sizes": sizes, "rank_single_set": single,
            "rank_kendall": tau, "sweep_iid_gaps": iid, "replay_roofline": replay_roof, "cpu_baseline": cpu,
            "e2e": e2e, "gpu_launches": launches, "clocks": clocks}
    for key, val in (("sweep_ase", ase), ("online_hazard", online), ("stale_snapshot", stale),
                     ("ablation", ablation)):
        if val is not None:
            line[key] = val
    if cpu is not None:
        cpu["rank"] = cpu_baseline_rank(rec, sigma)
    print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
