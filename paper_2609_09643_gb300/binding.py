"""Thin ctypes binding of include/unison.h (argument marshalling only).

Every computation runs in libunison.so's CUDA kernels; this module turns
numpy/torch objects into the C structs and pointers the ABI takes.  If the
library is missing the calls raise; there is no CPU path.
"""
from __future__ import annotations

import ctypes as C
import os
import threading
from typing import Iterable, List, Sequence

import numpy as np

from .native import LIB, LIB_DEBUG

POLICY = {"lru": 0, "timeout": 1, "spear": 2, "spear_tide": 3, "belady": 4, "lru_tide": 5}
FLAG_HAZARD_ONLINE = 1  # unison_replay_params.flags bit 0
FLAG_NO_GAP, FLAG_NO_HAZARD = 2, 4  # signal leave-one-out bits
STALE_SYNC = {"live": 0, "event": 1, "arrivals": 2, "gap_start": 3}  # UNISON_SYNC_*
KIND = ["COLD", "HIT_S", "HIT_H", "MISS", "PLACE_S", "PLACE_H", "BYPASS", "DEMOTE", "EVICT",
        "PROMOTE", "TIDE_DEMOTE", "EXPIRE"]
OK, ERR_ARG, ERR_IO, ERR_FORMAT, ERR_RANGE, ERR_CUDA, ERR_OOM, ERR_LOG_FULL, ERR_TIMEOUT, ERR_CAPACITY = \
    0, -1, -2, -3, -4, -5, -6, -7, -8, -9

DEFAULT_PARAMS = dict(
    policy="spear_tide", cap_fast_bytes=4 << 30, cap_hbm_bytes=64 << 30, kv_bytes_per_token=131072,
    max_sessions=0, ema_num=3, ema_den=10, hazard_bucket=1, ttl_us=10_000_000,
    penalty_q=500_000_000, dma_bytes_per_us=64_000, t_s_ps_per_tok=8192, t_h_ps_per_tok=32768,
    t_p_ps_per_tok=20_000_000, ttft_load=4,
)


class UnisonError(RuntimeError):
    def __init__(self, where: str, code: int):
        super().__init__(f"{where}: {strerror(code)} ({code})")
        self.code = code


class Turns(C.Structure):
    _fields_ = [("n_sessions", C.c_uint32), ("reserved", C.c_uint32), ("n_turns", C.c_uint64),
                ("turn_off", C.c_void_p), ("arrival_us", C.c_void_p), ("completion_us", C.c_void_p),
                ("in_tok", C.c_void_p), ("out_tok", C.c_void_p)]


class ReplayParams(C.Structure):
    _fields_ = [("policy", C.c_uint32), ("trace_idx", C.c_uint32), ("cap_fast_bytes", C.c_uint64),
                ("cap_hbm_bytes", C.c_uint64), ("kv_bytes_per_token", C.c_uint32),
                ("max_sessions", C.c_uint32), ("ema_num", C.c_uint32), ("ema_den", C.c_uint32),
                ("hazard_bucket", C.c_uint32), ("ttl_us", C.c_uint32), ("penalty_q", C.c_uint64),
                ("dma_bytes_per_us", C.c_uint64), ("t_s_ps_per_tok", C.c_uint64),
                ("t_h_ps_per_tok", C.c_uint64), ("t_p_ps_per_tok", C.c_uint64),
                ("ttft_load", C.c_uint32), ("flags", C.c_uint32), ("stale_sync", C.c_uint32),
                ("stale_m", C.c_uint32)]


RESULT_FIELDS = ["events", "req_warm", "cold", "hit_s", "hit_h", "miss", "bypass", "place_s", "place_h",
                 "evict", "demote", "promote", "tide_demote", "expire", "tok_hit_s", "tok_hit_h",
                 "tok_miss", "tok_computed", "tok_needed", "dma_bytes", "tide_calls",
                 "promoted_then_hit_s", "ttft_sum_lo", "ttft_sum_hi", "ttft_p50_ns", "ttft_n",
                 "decision_hash", "log_len", "vict_n", "vict_diff", "prom_n", "prom_diff"]


class ReplayResult(C.Structure):
    _fields_ = [(f, C.c_uint64) for f in RESULT_FIELDS] + [("status", C.c_int32), ("reserved", C.c_uint32)]


class Stats(C.Structure):
    _fields_ = [(f, C.c_double) for f in ("hit_rate", "amat_ps", "prered", "prefetch_acc", "ttft_mean_ns",
                                          "ttft_p50_ns")]


class Records(C.Structure):
    _fields_ = [("gap_q", C.c_void_p), ("last_ret", C.c_void_p), ("turn", C.c_void_p), ("kv_tok", C.c_void_p),
                ("tier", C.c_void_p), ("flags", C.c_void_p), ("n", C.c_uint64)]


class RankParams(C.Structure):
    _fields_ = [("sigma_q", C.c_uint16 * 51), ("reserved0", C.c_uint16), ("k", C.c_uint32),
                ("penalty_q", C.c_uint64), ("budget_bytes", C.c_uint64), ("kv_bytes_per_token", C.c_uint32),
                ("max_moves", C.c_uint32), ("free_fast_tok", C.c_uint64), ("free_hbm_tok", C.c_uint64)]


class RankOut(C.Structure):
    _fields_ = [("victims", C.c_void_p), ("promote", C.c_void_p), ("demote", C.c_void_p),
                ("counts", C.c_void_p), ("moved_bytes", C.c_void_p), ("keys", C.c_void_p)]


_lock = threading.Lock()
_lib = None

# Every symbol include/unison.h declares (checked by the ABI tests).
# the test library of native.build_debug() (include/unison_debug.h) adds these
DEBUG_EXPORTS = ["unison_debug_rank_wait_hooks"]
EXPORTS = ["unison_strerror", "unison_version", "unison_trace_create", "unison_trace_load",
           "unison_trace_upload", "unison_trace_free", "unison_trace_info", "unison_trace_device_bytes",
           "unison_replay_batch", "unison_stats", "unison_hazard_lut", "unison_rank_batch", "unison_rank",
           "unison_rank_cands_bytes", "unison_rank_shard", "unison_rank_merge",
           "unison_profile_enable", "unison_profile_read", "unison_launch_count",
           "unison_replay_batch_noalloc", "unison_ase", "unison_attainment", "unison_selftest_division",
           "unison_debug_fail_allocations"]


def lib_path() -> str:
    return LIB


def _bind_rank(L):
    L.unison_rank_batch.argtypes = [C.POINTER(Records), C.POINTER(RankParams), C.POINTER(RankOut), C.c_int,
                                    C.c_void_p]
    L.unison_rank.argtypes = [C.POINTER(Records), C.POINTER(RankParams), C.POINTER(RankOut), C.c_void_p]
    L.unison_rank_cands_bytes.argtypes = [C.c_uint32, C.c_uint32]
    L.unison_rank_cands_bytes.restype = C.c_uint64
    L.unison_rank_shard.argtypes = [C.POINTER(Records), C.c_uint64, C.POINTER(RankParams), C.c_void_p, C.c_void_p]
    L.unison_rank_merge.argtypes = [C.c_void_p, C.c_int, C.POINTER(RankParams), C.POINTER(RankOut), C.c_void_p]
    return L


_debug_lib = None


def debug_lib():
    """Load the ranking test library with its wait hooks (built by
    paper_2609_09643_gb300.native.build_debug()); pass it as ``lib_`` to
    RankCall."""
    global _debug_lib
    with _lock:
        if _debug_lib is None:
            if not os.path.exists(LIB_DEBUG):
                raise RuntimeError(f"{LIB_DEBUG} is missing: run native.build_debug() first")
            L = _bind_rank(C.CDLL(LIB_DEBUG))
            L.unison_debug_rank_wait_hooks.argtypes = [C.c_int, C.c_int]
            _debug_lib = L
    return _debug_lib


def lib():
    """Load libunison.so (built by paper_2609_09643_gb300.native.build())."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(LIB):
                raise RuntimeError(f"{LIB} is missing: run __graft_entry__.build() first")
            L = C.CDLL(LIB)
            L.unison_strerror.restype = C.c_char_p
            L.unison_strerror.argtypes = [C.c_int]
            L.unison_version.restype = C.c_int
            L.unison_trace_create.argtypes = [C.POINTER(Turns), C.POINTER(C.c_void_p)]
            L.unison_trace_load.argtypes = [C.c_char_p, C.POINTER(C.c_void_p)]
            L.unison_trace_upload.argtypes = [C.c_void_p, C.c_void_p]
            L.unison_trace_free.argtypes = [C.c_void_p]
            L.unison_trace_free.restype = None
            L.unison_trace_info.argtypes = [C.c_void_p, C.POINTER(C.c_uint32), C.POINTER(C.c_uint64),
                                            C.POINTER(C.c_uint64)]
            L.unison_trace_device_bytes.argtypes = [C.c_void_p]
            L.unison_trace_device_bytes.restype = C.c_uint64
            L.unison_replay_batch.argtypes = [C.POINTER(C.c_void_p), C.c_int, C.POINTER(ReplayParams), C.c_int,
                                              C.c_void_p, C.POINTER(ReplayResult), C.c_void_p, C.c_uint64,
                                              C.c_void_p]
            L.unison_stats.argtypes = [C.POINTER(ReplayResult), C.POINTER(ReplayParams), C.POINTER(Stats)]
            L.unison_hazard_lut.argtypes = [C.c_void_p, C.c_uint64, C.c_uint32, C.c_void_p, C.c_void_p,
                                            C.c_void_p]
            _bind_rank(L)
            L.unison_profile_enable.argtypes = [C.c_int]
            L.unison_profile_read.argtypes = [C.c_char_p, C.POINTER(C.c_double), C.POINTER(C.c_uint64), C.c_int]
            L.unison_launch_count.restype = C.c_uint64
            L.unison_replay_batch_noalloc.argtypes = L.unison_replay_batch.argtypes
            L.unison_ase.argtypes = [C.POINTER(Stats), C.c_int, C.c_int, C.POINTER(C.c_double)]
            L.unison_selftest_division.argtypes = [C.POINTER(C.c_uint64), C.c_void_p]
            L.unison_debug_fail_allocations.argtypes = [C.c_int]
            L.unison_debug_fail_allocations.restype = None
            L.unison_attainment.argtypes = [C.c_void_p, C.c_void_p, C.c_uint64, C.c_void_p, C.c_uint64,
                                            C.c_void_p, C.c_uint64, C.c_uint32, C.POINTER(AttainmentPoint)]
            _lib = L
    return _lib


def strerror(code: int) -> str:
    try:
        return lib().unison_strerror(code).decode()
    except RuntimeError:
        return f"status {code}"


def _check(where: str, rc: int, allow=(OK,)):
    if rc not in allow:
        raise UnisonError(where, rc)
    return rc


def _stream_handle(stream) -> int | None:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    return getattr(stream, "cuda_stream", stream)


# ------------------------------------------------------------------ traces --
class Trace:
    """Owner of a unison_trace handle built from host turn arrays (any object
    with turn_off, arrival_us, completion_us, in_tok, out_tok)."""

    def __init__(self, turns=None, path: str | None = None):
        h = C.c_void_p()
        if path is not None:
            _check("unison_trace_load", lib().unison_trace_load(path.encode(), C.byref(h)))
        else:
            arrs = (np.ascontiguousarray(turns.turn_off, np.uint64), np.ascontiguousarray(turns.arrival_us, np.uint64),
                    np.ascontiguousarray(turns.completion_us, np.uint64), np.ascontiguousarray(turns.in_tok, np.uint32),
                    np.ascontiguousarray(turns.out_tok, np.uint32))
            t = Turns(arrs[0].shape[0] - 1, 0, arrs[1].shape[0], *(a.ctypes.data for a in arrs))
            _check("unison_trace_create", lib().unison_trace_create(C.byref(t), C.byref(h)))
        self.handle = h
        self.uploaded = False

    def upload(self, stream=None) -> "Trace":
        _check("unison_trace_upload", lib().unison_trace_upload(self.handle, _stream_handle(stream)))
        self.uploaded = True
        return self

    def info(self):
        s, t, e = C.c_uint32(), C.c_uint64(), C.c_uint64()
        _check("unison_trace_info", lib().unison_trace_info(self.handle, C.byref(s), C.byref(t), C.byref(e)))
        return int(s.value), int(t.value), int(e.value)

    @property
    def device_bytes(self) -> int:
        return int(lib().unison_trace_device_bytes(self.handle))

    def close(self):
        if self.handle:
            lib().unison_trace_free(self.handle)
            self.handle = C.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def make_params(p: dict, trace_idx: int = 0) -> ReplayParams:
    q = dict(DEFAULT_PARAMS)
    q.update(p)
    pol = q["policy"]
    pol = POLICY[pol] if isinstance(pol, str) else int(pol)
    return ReplayParams(pol, q.get("trace_idx", trace_idx), q["cap_fast_bytes"], q["cap_hbm_bytes"],
                        q["kv_bytes_per_token"], q["max_sessions"], q["ema_num"], q["ema_den"],
                        q["hazard_bucket"], q["ttl_us"], q["penalty_q"], q["dma_bytes_per_us"],
                        q["t_s_ps_per_tok"], q["t_h_ps_per_tok"], q["t_p_ps_per_tok"], q["ttft_load"],
                        q.get("flags", (FLAG_HAZARD_ONLINE if q.get("hazard_online") else 0) |
                              (FLAG_NO_GAP if q.get("no_gap") else 0) | (FLAG_NO_HAZARD if q.get("no_hazard") else 0)),
                        STALE_SYNC[q.get("stale_sync", "live")] if isinstance(q.get("stale_sync", "live"), str)
                        else int(q["stale_sync"]), q.get("stale_m", 0))


def result_dict(r: ReplayResult) -> dict:
    d = {f: int(getattr(r, f)) for f in RESULT_FIELDS}
    d["status"] = int(r.status)
    d["ttft_sum"] = d["ttft_sum_lo"] + (d["ttft_sum_hi"] << 64)
    return d


def replay_batch(traces: Sequence[Trace], params: Sequence[dict], log_capacity: int = 0, stream=None,
                 results_dev=None, allow_status=(OK, ERR_LOG_FULL)):
    """Run unison_replay_batch.  Returns (list of result dicts, log) where log
    is a torch uint32 tensor [n_replays, log_capacity, 2] on the GPU or None."""
    import torch
    n = len(params)
    arr_t = (C.c_void_p * len(traces))(*(t.handle.value for t in traces))
    arr_p = (ReplayParams * n)(*(make_params(p) for p in params))
    out = (ReplayResult * n)()
    log = None
    if log_capacity:
        log = torch.zeros((n, log_capacity, 2), dtype=torch.int32, device="cuda")
    rc = lib().unison_replay_batch(arr_t, len(traces), arr_p, n,
                                   None if results_dev is None else results_dev.data_ptr(), out,
                                   None if log is None else log.data_ptr(), log_capacity, _stream_handle(stream))
    _check("unison_replay_batch", rc)
    res = [result_dict(out[i]) for i in range(n)]
    for i, r in enumerate(res):
        if r["status"] not in allow_status:
            raise UnisonError(f"replay {i}", r["status"])
    return res, log


def replay_batch_async(traces: Sequence[Trace], params: Sequence[dict], results_dev, stream=None, log=None,
                       log_capacity: int = 0):
    """Queue unison_replay_batch with device results only (no host sync)."""
    n = len(params)
    arr_t = (C.c_void_p * len(traces))(*(t.handle.value for t in traces))
    arr_p = (ReplayParams * n)(*(make_params(p) for p in params))
    rc = lib().unison_replay_batch(arr_t, len(traces), arr_p, n, results_dev.data_ptr(), None,
                                   None if log is None else log.data_ptr(), log_capacity, _stream_handle(stream))
    _check("unison_replay_batch", rc)


def results_from_tensor(t) -> List[dict]:
    """Decode a device/host uint8/int64 tensor holding unison_replay_result[n]."""
    b = t.detach().cpu().contiguous().view(-1).numpy().tobytes()
    sz = C.sizeof(ReplayResult)
    return [result_dict(ReplayResult.from_buffer_copy(b[i * sz:(i + 1) * sz])) for i in range(len(b) // sz)]


def result_nbytes(n: int) -> int:
    return n * C.sizeof(ReplayResult)


def decode_log(log_row, n: int):
    """(event, kind, session) numpy arrays of the first n decisions of one replay."""
    a = log_row[:n].cpu().numpy().astype(np.uint32)
    return a[:, 0].copy(), (a[:, 1] >> 24).astype(np.uint8), a[:, 1] & 0xFFFFFF


def stats(result: dict, params: dict) -> dict:
    r = ReplayResult(*[result[f] for f in RESULT_FIELDS], result.get("status", 0), 0)
    p = make_params(params)
    s = Stats()
    _check("unison_stats", lib().unison_stats(C.byref(r), C.byref(p), C.byref(s)))
    return {f: getattr(s, f) for f, _ in Stats._fields_}


def ase(stats_grid) -> List[float]:
    """unison_ase over stats_grid[config][dataset] (dicts as returned by
    stats(): hit_rate, amat_ps, ttft_mean_ns, ...): one value per config."""
    nc = len(stats_grid)
    nd = len(stats_grid[0]) if nc else 0
    arr = (Stats * (nc * nd))()
    for c, row in enumerate(stats_grid):
        if len(row) != nd:
            raise ValueError("every configuration needs the same datasets")
        for d, st in enumerate(row):
            arr[c * nd + d] = Stats(*[float(st.get(f, 0.0)) for f, _ in Stats._fields_])
    out = (C.c_double * max(nc, 1))()
    _check("unison_ase", lib().unison_ase(arr, nc, nd, out))
    return [out[i] for i in range(nc)]


class AttainmentPoint(C.Structure):
    _fields_ = [("sessions_seen", C.c_uint32), ("reserved", C.c_uint32), ("warm", C.c_uint64),
                ("hr_online", C.c_double), ("hr_offline", C.c_double), ("hr_lru", C.c_double),
                ("attainment", C.c_double)]


def attainment(trace: Trace, logs, n_points: int) -> List[dict]:
    """unison_attainment: logs are the (event, kind, session) arrays of the
    online-table, offline-table and LRU replays (decode_log output)."""
    packed = []
    for ev, kind, sess in logs:
        a = np.empty((len(ev), 2), dtype=np.uint32)
        a[:, 0] = ev
        a[:, 1] = (np.asarray(kind, np.uint32) << 24) | np.asarray(sess, np.uint32)
        packed.append(a)
    out = (AttainmentPoint * max(n_points, 1))()
    args = []
    for a in packed:
        args += [a.ctypes.data, a.shape[0]]
    _check("unison_attainment", lib().unison_attainment(trace.handle, *args, n_points, out))
    return [{f: getattr(out[i], f) for f, _ in AttainmentPoint._fields_ if f != "reserved"} for i in range(n_points)]


def selftest_division(stream=None) -> int:
    """unison_selftest_division: mismatches of the scores' multiply-high
    division against the quotient's definition (0 expected)."""
    out = C.c_uint64()
    _check("unison_selftest_division", lib().unison_selftest_division(C.byref(out), _stream_handle(stream)))
    return int(out.value)


def debug_fail_allocations(n: int) -> None:
    """The next n device allocations of the library fail as out of memory
    (fault injection for error-path tests; 0 clears)."""
    lib().unison_debug_fail_allocations(int(n))


def hazard_lut(turns_dev, bucket: int = 1, stream=None):
    """sigma_q[51] and h_q[51] (torch uint16-as-int16 tensors on the device)."""
    import torch
    sig = torch.zeros(51, dtype=torch.int16, device=turns_dev.device)
    hq = torch.zeros(51, dtype=torch.int16, device=turns_dev.device)
    _check("unison_hazard_lut", lib().unison_hazard_lut(turns_dev.data_ptr(), turns_dev.numel(), bucket,
                                                        sig.data_ptr(), hq.data_ptr(), _stream_handle(stream)))
    return sig, hq


# ------------------------------------------------------------ measurement --
def profile_enable(on: bool = True) -> None:
    _check("unison_profile_enable", lib().unison_profile_enable(1 if on else 0))


def profile_read(kernel: str, reset: bool = True):
    """(summed device ms, timed launches) of one kernel since the last reset."""
    ms, n = C.c_double(), C.c_uint64()
    _check("unison_profile_read", lib().unison_profile_read(kernel.encode(), C.byref(ms), C.byref(n),
                                                            1 if reset else 0))
    return float(ms.value), int(n.value)


def launch_count() -> int:
    return int(lib().unison_launch_count())


# ------------------------------------------------------- no-allocation path --
NOALLOC_SCRATCH_BYTES = 32 << 20


def replay_batch_noalloc(traces: Sequence[Trace], params: Sequence[dict], results_dev, stream=None, log=None,
                         log_capacity: int = 0) -> None:
    """unison_replay_batch_noalloc: the same replay, with the library's fixed
    device scratch instead of any allocation.  results_dev (and log, if
    given) are caller-owned device buffers; the call only marshals them."""
    n = len(params)
    arr_t = (C.c_void_p * len(traces))(*(t.handle.value for t in traces))
    arr_p = (ReplayParams * n)(*(make_params(p) for p in params))
    rc = lib().unison_replay_batch_noalloc(arr_t, len(traces), arr_p, n, results_dev.data_ptr(), None,
                                           None if log is None else log.data_ptr(), log_capacity,
                                           _stream_handle(stream))
    _check("unison_replay_batch_noalloc", rc)


# --------------------------------------------------------------- ranking --
def records_to_device(rec, device="cuda"):
    """Copy a synth.Records-like object (numpy SoA) to device tensors (bit
    patterns in signed torch dtypes)."""
    import torch
    conv = lambda a, dt: torch.from_numpy(np.ascontiguousarray(a).view(dt)).to(device)
    return dict(gap_q=conv(rec.gap_q.astype(np.uint32), np.int32), last_ret=conv(rec.last_ret.astype(np.uint32), np.int32),
                turn=conv(rec.turn.astype(np.uint16), np.int16), kv_tok=conv(rec.kv_tok.astype(np.uint32), np.int32),
                tier=conv(rec.tier.astype(np.uint8), np.uint8), flags=conv(rec.flags.astype(np.uint8), np.uint8))


def rank_outputs(n: int, k: int, max_moves: int, keys: bool = False, device="cuda"):
    import torch
    z = lambda m, dt: torch.zeros(max(m, 1), dtype=dt, device=device)
    return dict(victims=z(k, torch.int32), promote=z(max_moves, torch.int32), demote=z(max_moves, torch.int32),
                counts=z(4, torch.int32), moved=z(1, torch.int64), keys=z(n, torch.int64) if keys else None)


class RankCall:
    """The marshalled arguments of one unison_rank_batch call (ctypes arrays
    over the tensors' device pointers), reusable while those tensors live."""

    def __init__(self, sets: Sequence[dict], params: Sequence[dict], outs: Sequence[dict], lib_=None):
        n = len(sets)
        self.n = n
        self._lib = lib_
        self.rs = (Records * n)()
        self.ps = (RankParams * n)()
        self.os = (RankOut * n)()
        self._keep = (list(sets), list(outs))  # the pointers stay valid while these live
        for i, (r, p, o) in enumerate(zip(sets, params, outs)):
            self.rs[i] = _records(r)
            self.ps[i] = _rank_params(p)
            self.os[i] = _rank_out(o)

    def run(self, stream=None) -> None:
        L = self._lib if self._lib is not None else lib()
        _check("unison_rank_batch", L.unison_rank_batch(self.rs, self.ps, self.os, self.n, _stream_handle(stream)))

    def run_single(self, stream=None) -> None:
        """unison_rank on the one set this call holds."""
        assert self.n == 1
        L = self._lib if self._lib is not None else lib()
        _check("unison_rank", L.unison_rank(self.rs, self.ps, self.os, _stream_handle(stream)))


def rank_prepare(sets: Sequence[dict], params: Sequence[dict], outs: Sequence[dict]) -> RankCall:
    """Marshal a rank call once (see RankCall) for repeated launches."""
    return RankCall(sets, params, outs)


def rank(rec: dict, params: dict, out: dict, stream=None) -> None:
    """unison_rank: one device record set, one params dict, one output dict."""
    RankCall([rec], [params], [out]).run_single(stream)


def rank_batch(sets: Sequence[dict], params: Sequence[dict], outs: Sequence[dict], stream=None) -> None:
    """unison_rank_batch over device record sets; params per set: sigma_q[51],
    k, penalty_q, budget_bytes, kv_bytes_per_token, max_moves, free_fast_tok,
    free_hbm_tok."""
    RankCall(sets, params, outs).run(stream)


def _rank_params(p: dict) -> RankParams:
    sig = np.ascontiguousarray(np.asarray(p["sigma_q"], dtype=np.uint16))
    if sig.shape != (51,):
        raise ValueError("sigma_q must have 51 entries")
    return RankParams((C.c_uint16 * 51).from_buffer_copy(sig.tobytes()), 0, p.get("k", 0),
                      p.get("penalty_q", 500_000_000), p.get("budget_bytes", 0),
                      p.get("kv_bytes_per_token", 131072), p.get("max_moves", 0),
                      p.get("free_fast_tok", 0), p.get("free_hbm_tok", 0))


def _rank_out(o: dict) -> RankOut:
    return RankOut(o["victims"].data_ptr(), o["promote"].data_ptr(), o["demote"].data_ptr(),
                   o["counts"].data_ptr(), o["moved"].data_ptr(),
                   None if o.get("keys") is None else o["keys"].data_ptr())


def _records(r: dict) -> Records:
    return Records(r["gap_q"].data_ptr(), r["last_ret"].data_ptr(), r["turn"].data_ptr(), r["kv_tok"].data_ptr(),
                   r["tier"].data_ptr(), r["flags"].data_ptr(), r["gap_q"].numel())


def rank_cands_bytes(k: int, max_moves: int) -> int:
    """Bytes of one shard's candidate buffer (unison_rank_cands_bytes)."""
    return int(lib().unison_rank_cands_bytes(k, max_moves))


def rank_cands(k: int, max_moves: int, n_shards: int = 1, device="cuda"):
    """A uint8 device buffer for n_shards candidate buffers, back to back."""
    import torch
    return torch.zeros(n_shards * rank_cands_bytes(k, max_moves), dtype=torch.uint8, device=device)


def rank_shard(rec_slice: dict, index_offset: int, params: dict, cands, stream=None) -> None:
    """unison_rank_shard: rank records [index_offset, index_offset + n) of a
    live set (rec_slice: device arrays of the slice) into the uint8 device
    tensor cands (rank_cands_bytes(k, max_moves) bytes, 256-byte aligned)."""
    r, p = _records(rec_slice), _rank_params(params)
    _check("unison_rank_shard", lib().unison_rank_shard(C.byref(r), index_offset, C.byref(p), cands.data_ptr(),
                                                        _stream_handle(stream)))


def rank_merge(gathered, n_shards: int, params: dict, out: dict, stream=None) -> None:
    """unison_rank_merge over n_shards candidate buffers back to back in the
    uint8 device tensor gathered; writes out as unison_rank does."""
    p, o = _rank_params(params), _rank_out(out)
    _check("unison_rank_merge", lib().unison_rank_merge(gathered.data_ptr(), n_shards, C.byref(p), C.byref(o),
                                                        _stream_handle(stream)))


def rank_result(o: dict) -> dict:
    """Host copy of one set's outputs."""
    c = o["counts"].cpu().numpy().astype(np.uint32)
    res = dict(victims=o["victims"].cpu().numpy().astype(np.uint32)[: c[0]],
               promote=o["promote"].cpu().numpy().astype(np.uint32)[: c[1]],
               demote=o["demote"].cpu().numpy().astype(np.uint32)[: c[2]],
               moved_bytes=int(o["moved"].cpu().numpy().astype(np.uint64)[0]),
               status=int(c[3:4].view(np.int32)[0]))  # a status word: 0 or a negative UNISON_ERR_* code
    if o.get("keys") is not None:
        res["keys"] = o["keys"].cpu().numpy().view(np.uint64)
    return res
