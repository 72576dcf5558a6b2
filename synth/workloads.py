"""Workload definitions shared by the tests and the benchmark.

Parameters are written once in a neutral form and converted to the oracle's
and the library's argument names separately (the two share no code; this
module only renames keys and holds none of the method's arithmetic).
Tier costs (not given by the paper): t_s = kvB/16 ps per token (16 TB/s fast
tier), t_h = kvB/4 ps (4 TB/s), t_p = 20 us per prefill token; DMA 64 GB/s;
TTFT under 4x load.
"""
from __future__ import annotations

from .traces import paper_scale_trace, tiny_trace

GIB = 1 << 30
MIB = 1 << 20


def base(policy, cap_s, cap_h, kvb, **kw):
    p = dict(policy=policy, cap_s=cap_s, cap_h=cap_h, kvb=kvb, max_sessions=0, ema_num=3, ema_den=10,
             bucket=1, penalty=500_000_000, ttl=10_000_000, dma=64_000, load=4, t_p=20_000_000, online=False,
             stale="live", stale_m=0, no_gap=False, no_hazard=False)
    p.update(kw)
    return p


def to_oracle(p: dict) -> dict:
    return dict(policy=p["policy"], cap_s_bytes=p["cap_s"], cap_h_bytes=p["cap_h"], kv_bytes_per_token=p["kvb"],
                max_sessions=p["max_sessions"], ema_num=p["ema_num"], ema_den=p["ema_den"],
                hazard_bucket=p["bucket"], penalty_q=p["penalty"], ttl_us=p["ttl"], dma_bytes_per_us=p["dma"],
                ttft_load=p["load"], t_p_ps_per_tok=p["t_p"], hazard_online=bool(p.get("online")),
                stale_sync=p.get("stale", "live"), stale_m=p.get("stale_m", 0), no_gap=p.get("no_gap", False),
                no_hazard=p.get("no_hazard", False))


def to_lib(p: dict, trace_idx: int = 0) -> dict:
    kvb = p["kvb"]
    return dict(policy=p["policy"], trace_idx=trace_idx, cap_fast_bytes=p["cap_s"], cap_hbm_bytes=p["cap_h"],
                kv_bytes_per_token=kvb, max_sessions=p["max_sessions"], ema_num=p["ema_num"],
                ema_den=p["ema_den"], hazard_bucket=p["bucket"], penalty_q=p["penalty"], ttl_us=p["ttl"],
                dma_bytes_per_us=p["dma"], ttft_load=p["load"], t_p_ps_per_tok=p["t_p"],
                t_s_ps_per_tok=kvb // 16, t_h_ps_per_tok=kvb // 4, hazard_online=bool(p.get("online")),
                stale_sync=p.get("stale", "live"), stale_m=p.get("stale_m", 0), no_gap=p.get("no_gap", False),
                no_hazard=p.get("no_hazard", False))


# ---- the five workloads --------------------------------------------------------

def tiny_case():
    """64 sessions x 12 turns, 28,672 B/token, fast 512 MiB, HBM 8 GiB."""
    tr = tiny_trace(0)
    ps = [base(pol, 512 * MIB, 8 * GIB, 28672) for pol in ("lru", "spear", "spear_tide", "belady")]
    return tr, ps


KVB_PAPER = (28672, 131072, 163840)
POLICIES5 = ("lru", "timeout", "spear", "spear_tide", "belady")


def paper_scale_case():
    """Seed 1, 1,415 sessions / 33,596 turns; 5 policies x 2 gap mixes x 3 KV
    sizes = 30 replays at fast 4 GiB, HBM 64 GiB.  Returns ([traces], [(trace
    index, params)])."""
    trs = [paper_scale_trace(1, "coding"), paper_scale_trace(1, "general")]
    reps = [(ti, base(pol, 4 * GIB, 64 * GIB, kvb)) for ti in range(2) for kvb in KVB_PAPER for pol in POLICIES5]
    return trs, reps


def sweep_case(n_seeds: int = 8, gap_persist: float | None = None):
    """1,024 replays = 8 trace seeds x 8 capacity pairs x 16 (window, bucket)
    settings, SPEAR+TIDE at 131,072 B/token on the coding trace (gap_persist:
    the traces' gap persistence, None for the default)."""
    kw = {} if gap_persist is None else {"gap_persist": gap_persist}
    trs = [paper_scale_trace(seed, "coding", **kw) for seed in range(n_seeds)]
    reps = []
    for ti in range(n_seeds):
        for cs in (1, 2, 4, 8):
            for ch in (32, 128):
                for w in (4, 8, 16, 32):
                    for b in (1, 2, 4, 8):
                        reps.append((ti, base("spear_tide", cs * GIB, ch * GIB, 131072, ema_num=2,
                                              ema_den=w + 1, bucket=b)))
    return trs, reps


def large_pool_params():
    return base("spear_tide", 16 * GIB, 160 * GIB, 163840)
