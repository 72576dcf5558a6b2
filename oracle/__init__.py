"""CPU oracle for the UNISON hot path -- TEST INFRASTRUCTURE ONLY.

A ctypes wrapper over ``unison_oracle.c``: a plain, single-threaded C
restatement of the paper's SPEAR score (Sec. III-B and eqs. uq, hq, survq,
gapq, t1, t2, scoreq, ema-int of Sec. IV-C), the TIDE fill (Sec. III-C) and
the joint event loop (Algorithm 1), plus the standalone ranking of a live
set.  Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  It shares no code with the CUDA
library; the two meet only in the seeded inputs of the ``synth`` package.

Replay parameters are passed as a plain dict with the keys of
``DEFAULT_PARAMS``.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "unison_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB = os.path.join(_BUILD, "libunison_oracle.so")

POLICIES = {"lru": 0, "timeout": 1, "spear": 2, "spear_tide": 3, "belady": 4, "lru_tide": 5}
# R28 sync points of the stale-snapshot (dual design) replays
STALE_SYNC = {"live": 0, "event": 1, "arrivals": 2, "gap_start": 3}
KINDS = ["COLD", "HIT_S", "HIT_H", "MISS", "PLACE_S", "PLACE_H", "BYPASS", "DEMOTE", "EVICT",
         "PROMOTE", "TIDE_DEMOTE", "EXPIRE"]

DEFAULT_PARAMS = dict(
    policy="spear_tide", cap_s_bytes=4 << 30, cap_h_bytes=64 << 30, kv_bytes_per_token=131072,
    max_sessions=0, ema_num=3, ema_den=10, hazard_bucket=1, penalty_q=500_000_000,
    ttl_us=10_000_000, dma_bytes_per_us=64_000, t_s_ps_per_tok=8192, t_h_ps_per_tok=32768,
    t_p_ps_per_tok=20_000_000, ttft_load=4,
)


class _Trace(C.Structure):
    _fields_ = [("n_sessions", C.c_uint32), ("pad0", C.c_uint32), ("n_turns", C.c_uint64),
                ("turn_off", C.c_void_p), ("arrival_us", C.c_void_p),
                ("completion_us", C.c_void_p), ("in_tok", C.c_void_p), ("out_tok", C.c_void_p)]


class _Params(C.Structure):
    _fields_ = [("policy", C.c_uint32), ("hazard_bucket", C.c_uint32),
                ("cap_s_bytes", C.c_uint64), ("cap_h_bytes", C.c_uint64),
                ("kv_bytes_per_token", C.c_uint32), ("max_sessions", C.c_uint32),
                ("ema_num", C.c_uint32), ("ema_den", C.c_uint32), ("penalty_q", C.c_uint64),
                ("ttl_us", C.c_uint32), ("ttft_load", C.c_uint32),
                ("dma_bytes_per_us", C.c_uint64), ("prefill_ns_per_tok", C.c_uint64),
                ("debug", C.c_uint32), ("hazard_online", C.c_uint32), ("stale_sync", C.c_uint32),
                ("stale_m", C.c_uint32), ("signals", C.c_uint32), ("pad3", C.c_uint32)]


RESULT_FIELDS = ["events", "req_warm", "cold", "hit_s", "hit_h", "miss", "bypass", "place_s",
                 "place_h", "evict", "demote", "promote", "tide_demote", "expire", "tok_hit_s",
                 "tok_hit_h", "tok_miss", "tok_computed", "tok_needed", "dma_bytes", "tide_calls",
                 "promoted_then_hit_s", "ttft_sum_lo", "ttft_sum_hi", "ttft_p50_ns", "ttft_n",
                 "decision_hash", "log_len", "vict_n", "vict_diff", "prom_n", "prom_diff"]


class _Result(C.Structure):
    _fields_ = [(f, C.c_uint64) for f in RESULT_FIELDS] + [("status", C.c_int32), ("pad2", C.c_uint32)]


class _Records(C.Structure):
    _fields_ = [("gap_q", C.c_void_p), ("last_ret", C.c_void_p), ("turn", C.c_void_p),
                ("kv_tok", C.c_void_p), ("tier", C.c_void_p), ("flags", C.c_void_p),
                ("n", C.c_uint64)]


_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc into ``oracle/_build`` (portable C, no -march)."""
    os.makedirs(_BUILD, exist_ok=True)
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=gnu11", "-ffp-contract=off", "-fPIC", "-shared",
                               "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


def _bind(L):
    """Declare the argument and result types of the oracle's entry points."""
    L.or_replay.argtypes = [C.POINTER(_Trace), C.POINTER(_Params), C.POINTER(_Result),
                            C.c_void_p, C.c_uint64, C.c_void_p]
    L.or_replay.restype = C.c_int
    L.or_hazard_lut.argtypes = [C.c_void_p, C.c_uint64, C.c_uint32, C.c_void_p, C.c_void_p]
    L.or_hazard_lut.restype = C.c_int
    L.or_spear_score.argtypes = [C.c_uint64, C.c_uint32, C.c_uint64, C.c_int]
    L.or_spear_score.restype = C.c_uint64
    L.or_ema.argtypes = [C.c_uint64, C.c_uint64, C.c_uint32, C.c_uint32]
    L.or_ema.restype = C.c_uint64
    L.or_rank.argtypes = ([C.POINTER(_Records), C.c_void_p, C.c_uint64, C.c_uint32,
                           C.c_uint64, C.c_uint32, C.c_uint64, C.c_uint64]
                          + [C.c_void_p] * 8 + [C.c_uint32])
    L.or_rank.restype = C.c_int
    L.or_kendall_brute.argtypes = [C.c_void_p, C.c_void_p, C.c_uint64]
    L.or_kendall_brute.restype = C.c_double
    L.or_ase.argtypes = [C.c_void_p, C.c_void_p, C.c_void_p, C.c_int, C.c_int, C.c_void_p]
    L.or_ase.restype = None
    L.or_attainment.argtypes = [C.POINTER(_Trace), C.c_void_p, C.c_void_p, C.c_uint32, C.c_void_p]
    L.or_attainment.restype = C.c_int
    return L


def lib():
    global _lib
    with _lock:
        if _lib is None:
            _lib = _bind(C.CDLL(build()))
    return _lib


def build_variant(source: str, out_dir: str):
    """Compile a modified copy of the oracle's C source (a test plants one
    mistake in it to show that a pin catches that mistake) and load it.  The
    result is passed as ``lib_`` to ``replay``."""
    src = os.path.join(out_dir, "variant.c")
    so = os.path.join(out_dir, "libvariant.so")
    with open(src, "w") as f:
        f.write(source)
    subprocess.check_call(["gcc", "-O1", "-std=gnu11", "-ffp-contract=off", "-fPIC", "-shared", "-o", so, src,
                           "-lm"])
    return _bind(C.CDLL(so))


def source() -> str:
    """The oracle's C source text."""
    with open(_SRC) as f:
        return f.read()


def _ptr(a: np.ndarray) -> int:
    return a.ctypes.data


def _trace_struct(tr):
    arrs = (np.ascontiguousarray(tr.turn_off, np.uint64), np.ascontiguousarray(tr.arrival_us, np.uint64),
            np.ascontiguousarray(tr.completion_us, np.uint64), np.ascontiguousarray(tr.in_tok, np.uint32),
            np.ascontiguousarray(tr.out_tok, np.uint32))
    s = _Trace(tr.n_sessions, 0, tr.n_turns, *(_ptr(a) for a in arrs))
    return s, arrs


def _params_struct(p: dict, debug: bool):
    q = dict(DEFAULT_PARAMS)
    q.update(p)
    pol = q["policy"]
    pol = POLICIES[pol] if isinstance(pol, str) else int(pol)
    return _Params(pol, q["hazard_bucket"], q["cap_s_bytes"], q["cap_h_bytes"],
                   q["kv_bytes_per_token"], q["max_sessions"], q["ema_num"], q["ema_den"],
                   q["penalty_q"], q["ttl_us"], q["ttft_load"], q["dma_bytes_per_us"],
                   q["t_p_ps_per_tok"] // 1000, 1 if debug else 0, 1 if q.get("hazard_online") else 0,
                   STALE_SYNC[q.get("stale_sync", "live")], q.get("stale_m", 0),
                   (2 if q.get("no_gap") else 0) | (4 if q.get("no_hazard") else 0), 0)


def replay(tr, params: dict, log: bool = False, ttft: bool = False, debug: bool = False,
           log_capacity: int | None = None, lib_=None) -> dict:
    """Replay one trace under one policy; returns the counters (and, on
    request, the decision log as (event, kind, session) arrays and the
    per-request TTFT values in ns).  ``lib_``: a library from
    ``build_variant`` instead of the oracle itself."""
    L = lib_ if lib_ is not None else lib()
    ts, keep = _trace_struct(tr)
    ps = _params_struct(params, debug)
    res = _Result()
    cap = (log_capacity if log_capacity is not None else 16 * tr.n_events + 16) if log else 0
    logbuf = np.zeros(2 * cap, dtype=np.uint32) if log else None
    tt = np.zeros(tr.n_turns + 1, dtype=np.uint64) if ttft else None
    L.or_replay(C.byref(ts), C.byref(ps), C.byref(res), _ptr(logbuf) if log else None, cap,
                _ptr(tt) if ttft else None)
    out = {f: int(getattr(res, f)) for f in RESULT_FIELDS}
    out["status"] = int(res.status)
    out["ttft_sum"] = out["ttft_sum_lo"] + (out["ttft_sum_hi"] << 64)
    if log:
        n = min(out["log_len"], cap)
        lb = logbuf[: 2 * n].reshape(-1, 2)
        out["log"] = (lb[:, 0].copy(), (lb[:, 1] >> 24).astype(np.uint8), lb[:, 1] & 0xFFFFFF)
    if ttft:
        out["ttft"] = tt[: out["ttft_n"]].copy()
    return out


def hazard_lut(turns_per_session, bucket: int = 1):
    """(h_q[51], sigma_q[51]) of eqs. (hazard), (hq), (survq) for bucket width w."""
    t = np.ascontiguousarray(turns_per_session, dtype=np.uint32)
    h = np.zeros(51, dtype=np.uint16)
    s = np.zeros(51, dtype=np.uint16)
    rc = lib().or_hazard_lut(_ptr(t), t.shape[0], bucket, _ptr(h), _ptr(s))
    if rc != 0:
        raise ValueError(f"or_hazard_lut: {rc}")
    return h, s


def spear_score(g_q: int, sigma_q: int, penalty_q: int = 500_000_000, done: bool = False) -> int:
    return int(lib().or_spear_score(g_q, sigma_q, penalty_q, 1 if done else 0))


def ema(g_q: int, g_new: int, a_num: int = 3, a_den: int = 10) -> int:
    return int(lib().or_ema(g_q, g_new, a_num, a_den))


def rank(rec, sigma_q51, penalty_q: int, k: int, budget_bytes: int, kv_bytes_per_token: int,
         free_s_tok: int, free_h_tok: int, keys: bool = False, max_moves: int = 1 << 16) -> dict:
    """Keys, top-k victims and the TIDE fill of one live set (see or_rank)."""
    arrs = [np.ascontiguousarray(a) for a in (rec.gap_q.astype(np.uint32), rec.last_ret.astype(np.uint32),
                                               rec.turn.astype(np.uint16), rec.kv_tok.astype(np.uint32),
                                               rec.tier.astype(np.uint8), rec.flags.astype(np.uint8))]
    rs = _Records(*(_ptr(a) for a in arrs), rec.n)
    sig = np.ascontiguousarray(sigma_q51, dtype=np.uint16)
    vic = np.zeros(max(k, 1), dtype=np.uint32)
    pro = np.zeros(max_moves, dtype=np.uint32)
    dem = np.zeros(max_moves, dtype=np.uint32)
    nv, npro, ndem = C.c_uint32(), C.c_uint32(), C.c_uint32()
    moved = C.c_uint64()
    kk = np.zeros(rec.n, dtype=np.uint64) if keys else None
    rc = lib().or_rank(C.byref(rs), _ptr(sig), penalty_q, k, budget_bytes, kv_bytes_per_token,
                       free_s_tok, free_h_tok, _ptr(vic), C.addressof(nv), _ptr(pro),
                       C.addressof(npro), _ptr(dem), C.addressof(ndem), C.addressof(moved),
                       _ptr(kk) if keys else None, max_moves)
    if rc != 0:
        raise RuntimeError(f"or_rank: {rc}")
    out = dict(victims=vic[: nv.value].copy(), promote=pro[: npro.value].copy(),
               demote=dem[: ndem.value].copy(), moved_bytes=int(moved.value))
    if keys:
        out["keys"] = kk
    return out


def kendall_brute(x, y) -> float:
    a = np.ascontiguousarray(x, dtype=np.float64)
    b = np.ascontiguousarray(y, dtype=np.float64)
    return float(lib().or_kendall_brute(_ptr(a), _ptr(b), a.shape[0]))


def ase(hit_rate, amat, ttft):
    """Eq. (ase) per configuration: arrays [n_configs][n_datasets] of HR,
    AMAT and TTFT; returns n_configs values."""
    hr = np.ascontiguousarray(hit_rate, dtype=np.float64)
    am = np.ascontiguousarray(amat, dtype=np.float64)
    tt = np.ascontiguousarray(ttft, dtype=np.float64)
    nc, nd = hr.shape
    out = np.zeros(nc, dtype=np.float64)
    lib().or_ase(_ptr(hr), _ptr(am), _ptr(tt), nc, nd, _ptr(out))
    return out


def attainment(tr, logs, n_points: int):
    """Eq. (attainment) over the windows of reading R27: ``logs`` are the
    (event, kind, session) triples of the online-table, offline-table and LRU
    replays (``replay(..., log=True)["log"]``).  Returns (status, array
    [n_points, 6] of n_j, warm requests, H_on, H_off, H_LRU, A_j)."""
    ts, keep = _trace_struct(tr)
    packed = []
    for ev, kind, sess in logs:
        a = np.empty((len(ev), 2), dtype=np.uint32)
        a[:, 0] = ev
        a[:, 1] = (np.asarray(kind, np.uint32) << 24) | np.asarray(sess, np.uint32)
        packed.append(a)
    ptrs = (C.c_void_p * 3)(*(_ptr(a) for a in packed))
    lens = np.array([a.shape[0] for a in packed], dtype=np.uint64)
    out = np.zeros((max(n_points, 1), 6), dtype=np.float64)
    rc = lib().or_attainment(C.byref(ts), C.cast(ptrs, C.c_void_p), _ptr(lens), n_points, _ptr(out))
    return rc, out[:n_points]
