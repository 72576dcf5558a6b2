"""Seeded synthetic agent-session traces.

The paper's SWE-bench/GAIA traces (1,415 sessions, 33,596 turns) are not
available, so these generators stand in for them with the same shapes:
sessions of T_s turns, lognormal tool-wait gaps, a prefix that grows every
turn, and Poisson session starts.  A trace is only turn records
(arrival time, completion time, tokens in, tokens out); building events,
hazard tables, scores and decisions from it is left to the code under test.

Workload model (one reading, stated once, used by every generator here):

* session s starts at ``a_{s,0}``; starts are cumulative exponential
  inter-arrival draws rounded to whole microseconds, so session ids
  0..S-1 are in order of first arrival;
* turn k needs ``in_k`` tokens and leaves ``out_k = in_k + decode_k``
  resident, with ``in_0 = 2048``, ``in_k = out_{k-1} + insert_k``,
  ``insert_k ~ round(LN(400, 0.8))`` (at least 1) and
  ``decode_k ~ U{64..256}``;
* the trace is open loop: ``c_{s,k} = a_{s,k} + 20 us * decode_k`` and
  ``a_{s,k+1} = c_{s,k} + gap``, the gap drawn from a lognormal mixture and
  clamped to [1, 2**31 - 1] microseconds;
* gaps recur per session (the gap average of Sec. IV-C tracks a session's
  characteristic return interval): a session draws its mixture component
  once and a characteristic interval ``med * exp(sig * sqrt(rho) * Z_s)``,
  and each gap is that interval times ``exp(sig * sqrt(1 - rho) * Z_{s,k})``:
  each component keeps its marginal LN(med, sig), and log-gaps of one
  session correlate with coefficient ``rho`` (0.7; 0 draws every gap on its
  own, component included).

Times are absolute unsigned 64-bit microseconds.
"""
from __future__ import annotations

import dataclasses
import struct
from typing import Sequence, Tuple

import numpy as np

from . import rng

# (weight, median seconds, sigma) components of the tool-wait gap mixtures.
GAP_MIX_CONFIG0: Tuple[Tuple[float, float, float], ...] = ((1.0, 3.0, 1.2),)
GAP_MIX_CODING = ((0.7, 1.5, 1.2), (0.3, 30.0, 1.2))
GAP_MIX_GENERAL = ((0.5, 4.0, 1.2), (0.5, 90.0, 1.2))

FIRST_PREFIX_TOKENS = 2048
DECODE_US_PER_TOKEN = 20
GAP_MAX_US = (1 << 31) - 1

# Share of a gap's log-variance fixed per session.
GAP_PERSIST = 0.7

# Stream ids: one counter-addressed stream per kind of draw.
_ST_START, _ST_TURNS, _ST_DECODE, _ST_INSERT, _ST_GAPC, _ST_GAPN = 1, 2, 4, 6, 8, 10
_ST_SESSC, _ST_SESSN = 12, 14  # per-session component and interval (by session id)

_UTR_MAGIC = b"UTR1"


@dataclasses.dataclass
class Trace:
    """Turn records of one trace, session-major (CSR by ``turn_off``)."""

    turn_off: np.ndarray       # uint64[S + 1]
    arrival_us: np.ndarray     # uint64[T]
    completion_us: np.ndarray  # uint64[T]
    in_tok: np.ndarray         # uint32[T]
    out_tok: np.ndarray        # uint32[T]

    @property
    def n_sessions(self) -> int:
        return int(self.turn_off.shape[0] - 1)

    @property
    def n_turns(self) -> int:
        return int(self.arrival_us.shape[0])

    @property
    def n_events(self) -> int:
        return 2 * self.n_turns

    def turns_per_session(self) -> np.ndarray:
        return np.diff(self.turn_off).astype(np.int64)

    def contiguous(self) -> "Trace":
        return Trace(*(np.ascontiguousarray(a) for a in (
            self.turn_off.astype(np.uint64), self.arrival_us.astype(np.uint64),
            self.completion_us.astype(np.uint64), self.in_tok.astype(np.uint32),
            self.out_tok.astype(np.uint32))))


def geometric_turns(seed: int, n_sessions: int, mean: float, lo: int, hi: int,
                    total: int | None = None) -> np.ndarray:
    """Turns per session: Geometric(p = 1/mean) on {1, 2, ...} conditioned on
    [lo, hi], drawn by inversion; optionally nudged by +-1 round-robin over
    session ids (within the bounds) until the turns sum to ``total``."""
    p = 1.0 / mean
    q = 1.0 - p
    m = hi - lo + 1
    u = rng.uniform(seed, _ST_TURNS, np.arange(n_sessions))
    j = np.floor(np.log1p(-u * (1.0 - q ** m)) / np.log(q)).astype(np.int64)
    t = lo + np.clip(j, 0, m - 1)
    if total is not None:
        diff = int(total - t.sum())
        if diff != 0 and not (lo * n_sessions <= total <= hi * n_sessions):
            raise ValueError("turn total outside the bounds")
        s = 0
        while diff != 0:
            if diff > 0 and t[s] < hi:
                t[s] += 1
                diff -= 1
            elif diff < 0 and t[s] > lo:
                t[s] -= 1
                diff += 1
            s = (s + 1) % n_sessions
    return t


def _lognormal_mixture(seed: int, sess: np.ndarray, idx: np.ndarray, mix, rho: float) -> np.ndarray:
    """Seconds drawn from a lognormal mixture (see module doc): the component
    by one uniform (per session when rho > 0, else per turn), then median *
    exp(sigma * (sqrt(rho) Z_s + sqrt(1 - rho) Z_{s,k}))."""
    if not 0.0 <= rho <= 1.0:
        raise ValueError("gap persistence must be in [0, 1]")
    su = sess.astype(np.uint64)
    u = rng.uniform(seed, _ST_SESSC, su) if rho > 0 else rng.uniform(seed, _ST_GAPC, idx)
    z = np.sqrt(1.0 - rho) * rng.normal(seed, _ST_GAPN, idx)
    if rho > 0:
        z = z + np.sqrt(rho) * rng.normal(seed, _ST_SESSN, su)
    out = np.empty(idx.shape[0], dtype=np.float64)
    acc = 0.0
    chosen = np.zeros(idx.shape[0], dtype=bool)
    for i, (w, med, sig) in enumerate(mix):
        acc += w
        sel = (~chosen) & ((u < acc) | (i == len(mix) - 1))
        out[sel] = med * np.exp(sig * z[sel])
        chosen |= sel
    return out


def make_trace(seed: int, turns: Sequence[int] | np.ndarray, start_mean_s: float,
               gap_mix=GAP_MIX_CODING, first_start_at_zero: bool = False,
               gap_persist: float = GAP_PERSIST) -> Trace:
    """Build a trace with the given turns per session (see module doc)."""
    t_s = np.asarray(turns, dtype=np.int64)
    n = t_s.shape[0]
    if n == 0:
        z64 = np.zeros(0, dtype=np.uint64)
        return Trace(np.zeros(1, np.uint64), z64, z64.copy(), np.zeros(0, np.uint32),
                     np.zeros(0, np.uint32))
    if t_s.min() < 1 or t_s.max() >= (1 << 16):
        raise ValueError("turns per session must be in [1, 65535]")
    inter = np.floor(rng.exponential(seed, _ST_START, np.arange(n), start_mean_s * 1e6) + 0.5)
    inter = inter.astype(np.uint64)
    if first_start_at_zero:
        inter[0] = 0
    start = np.cumsum(inter, dtype=np.uint64)

    off = np.zeros(n + 1, dtype=np.uint64)
    off[1:] = np.cumsum(t_s).astype(np.uint64)
    total = int(off[-1])
    sess = np.repeat(np.arange(n, dtype=np.int64), t_s)
    k = np.arange(total, dtype=np.int64) - off[:-1].astype(np.int64)[sess]
    addr = (sess.astype(np.uint64) << np.uint64(16)) | k.astype(np.uint64)

    decode = rng.randint(seed, _ST_DECODE, addr, 64, 256)
    ins = np.floor(400.0 * np.exp(0.8 * rng.normal(seed, _ST_INSERT, addr)) + 0.5)
    ins = np.maximum(ins, 1.0).astype(np.int64)
    ins[k == 0] = FIRST_PREFIX_TOKENS  # turn 0 brings the first prefix
    # in_k = out_{k-1} + insert_k and out_k = in_k + decode_k, so
    # in_k = sum_{j<=k} insert_j + sum_{j<k} decode_j  (per session).
    step = ins + decode
    cum = np.cumsum(step)
    base = np.concatenate(([0], cum))[off[:-1].astype(np.int64)][sess]
    out_tok = cum - base
    in_tok = out_tok - decode
    if out_tok.max(initial=0) >= (1 << 32):
        raise ValueError("token counts overflow 32 bits")

    gap = np.floor(_lognormal_mixture(seed, sess, addr, gap_mix, gap_persist) * 1e6 + 0.5)
    gap = np.clip(gap, 1, GAP_MAX_US).astype(np.int64)
    gap[k == 0] = 0  # turn 0 has no preceding gap
    # a_k = start + sum_{j<k} (20 us * decode_j) + sum_{j<=k} gap_j
    adv = gap + np.concatenate(([0], DECODE_US_PER_TOKEN * decode[:-1]))
    adv[k == 0] = 0
    cadv = np.cumsum(adv)
    abase = cadv[off[:-1].astype(np.int64)][sess]
    arrival = start[sess] + (cadv - abase).astype(np.uint64)
    completion = arrival + (DECODE_US_PER_TOKEN * decode).astype(np.uint64)
    return Trace(off, arrival.astype(np.uint64), completion.astype(np.uint64),
                 in_tok.astype(np.uint32), out_tok.astype(np.uint32))


# ---- the workload shapes -----------------------------------------------------

def tiny_trace(seed: int = 0) -> Trace:
    """64 sessions x 12 turns, starts Poisson with mean 2 s, gaps LN(3 s, 1.2)."""
    return make_trace(seed, np.full(64, 12), 2.0, GAP_MIX_CONFIG0)


def paper_scale_trace(seed: int = 1, mix: str = "coding", gap_persist: float = GAP_PERSIST) -> Trace:
    """1,415 sessions / 33,596 turns, T_s ~ Geometric(mean 23.7) on [2, 200]
    adjusted to the exact total, starts Poisson with mean 2 s.  gap_persist 0
    draws every gap's component and value independently."""
    gm = {"coding": GAP_MIX_CODING, "general": GAP_MIX_GENERAL}[mix]
    t = geometric_turns(seed, 1415, 23.7, 2, 200, total=33596)
    return make_trace(seed, t, 2.0, gm, gap_persist=gap_persist)


def large_pool_trace(seed: int, n_sessions: int = 65536) -> Trace:
    """65,536 sessions, T_s ~ Geometric(mean 24) on [2, 200], starts Poisson
    with mean 1 ms (so nearly every session is live at once), general mix."""
    t = geometric_turns(seed, n_sessions, 24.0, 2, 200)
    return make_trace(seed, t, 1e-3, GAP_MIX_GENERAL)


def bimodal_trace(seed: int = 7, n_sessions: int = 96) -> Trace:
    """Half the sessions run 4 turns and half run 40, so the turn-indexed
    hazard is far from constant (a workload that exercises the hazard term)."""
    t = np.where(rng.uniform(seed, 99, np.arange(n_sessions)) < 0.5, 4, 40)
    return make_trace(seed, t, 1.0, GAP_MIX_CODING)


def trace_from_turns(arrivals: Sequence[Sequence[int]], completions: Sequence[Sequence[int]],
                     in_tok: Sequence[Sequence[int]], out_tok: Sequence[Sequence[int]]) -> Trace:
    """Hand-written trace from per-session turn lists (small test cases)."""
    n = len(arrivals)
    off = np.zeros(n + 1, dtype=np.uint64)
    off[1:] = np.cumsum([len(a) for a in arrivals]).astype(np.uint64)
    cat = lambda xs, dt: np.array([v for x in xs for v in x], dtype=dt)
    return Trace(off, cat(arrivals, np.uint64), cat(completions, np.uint64),
                 cat(in_tok, np.uint32), cat(out_tok, np.uint32))


# ---- .utr file format -------------------------------------------------------
# little endian: "UTR1", u32 n_sessions, u64 n_turns, then u64 turn_off[S+1],
# u64 arrival_us[T], u64 completion_us[T], u32 in_tok[T], u32 out_tok[T].

def save_utr(tr: Trace, path: str) -> None:
    tr = tr.contiguous()
    with open(path, "wb") as f:
        f.write(_UTR_MAGIC + struct.pack("<IQ", tr.n_sessions, tr.n_turns))
        for a in (tr.turn_off, tr.arrival_us, tr.completion_us, tr.in_tok, tr.out_tok):
            f.write(a.astype(a.dtype.newbyteorder("<")).tobytes())


def load_utr(path: str) -> Trace:
    with open(path, "rb") as f:
        head = f.read(16)
        if head[:4] != _UTR_MAGIC:
            raise ValueError("not a .utr trace")
        s, t = struct.unpack("<IQ", head[4:])
        rd = lambda dt, n: np.frombuffer(f.read(n * np.dtype(dt).itemsize), dtype=dt).copy()
        return Trace(rd("<u8", s + 1).astype(np.uint64), rd("<u8", t).astype(np.uint64),
                     rd("<u8", t).astype(np.uint64), rd("<u4", t).astype(np.uint32),
                     rd("<u4", t).astype(np.uint32))
