"""Seeded live-set records for the standalone ranking workload.

One record per live session, structure of arrays, drawn so that each field
looks like a session of the paper-scale coding workload caught at a random
moment:

* ``turn``: T_s ~ Geometric(mean 23.7) on [2, 200], t ~ U{0..T_s-1};
* ``flags``: bit0 pinned (mid-turn) with probability 1/64; otherwise bit1
  done when t is the session's last turn;
* ``gap_q``: 0 before the first gap (t = 0), otherwise one draw of the
  coding gap mixture in microseconds (a stand-in for the session's gap
  average, drawn directly rather than computed);
* ``kv_tok``: 2048 + t * LN(545, 0.3) + U{64..256} resident tokens
  (monotone prefix growth at the coding trace's mean growth per turn);
* ``tier``: 1 (fast tier) with probability 1/16, else 2 (HBM tier);
* ``last_ret``: 2**31 - U[0, 2**30) microseconds.
"""
from __future__ import annotations

import dataclasses

import numpy as np

from . import rng
from .traces import GAP_MIX_CODING, GAP_MAX_US, _lognormal_mixture

TIER_S, TIER_H = 1, 2
FLAG_PINNED, FLAG_DONE = 1, 2

_R_TURNS, _R_T, _R_PIN, _R_GAP, _R_KV, _R_DEC, _R_TIER, _R_RET = 21, 22, 23, 24, 26, 28, 29, 30


@dataclasses.dataclass
class Records:
    gap_q: np.ndarray     # uint32[N]  (non-negative int32 range)
    last_ret: np.ndarray  # uint32[N]
    turn: np.ndarray      # uint16[N]
    kv_tok: np.ndarray    # uint32[N]
    tier: np.ndarray      # uint8[N]
    flags: np.ndarray     # uint8[N]

    @property
    def n(self) -> int:
        return int(self.gap_q.shape[0])


def make_records(seed: int, n: int) -> Records:
    i = np.arange(n, dtype=np.uint64)
    p = 1.0 / 23.7
    q = 1.0 - p
    m = 199
    u = rng.uniform(seed, _R_TURNS, i)
    t_s = 2 + np.clip(np.floor(np.log1p(-u * (1.0 - q ** m)) / np.log(q)), 0, m - 1).astype(np.int64)
    t = np.minimum(np.floor(rng.uniform(seed, _R_T, i) * t_s).astype(np.int64), t_s - 1)
    pinned = rng.uniform(seed, _R_PIN, i) < (1.0 / 64.0)
    done = (~pinned) & (t == t_s - 1)
    flags = (pinned.astype(np.uint8) * FLAG_PINNED) | (done.astype(np.uint8) * FLAG_DONE)
    gap = np.floor(_lognormal_mixture(seed ^ 0x5A5A, i, i, GAP_MIX_CODING, 0.0) * 1e6 + 0.5)
    gap = np.clip(gap, 1, GAP_MAX_US).astype(np.int64)
    gap[t == 0] = 0
    growth = 545.0 * np.exp(0.3 * rng.normal(seed, _R_KV, i))
    kv = 2048 + np.floor(t * growth + 0.5).astype(np.int64) + rng.randint(seed, _R_DEC, i, 64, 256)
    tier = np.where(rng.uniform(seed, _R_TIER, i) < (1.0 / 16.0), TIER_S, TIER_H).astype(np.uint8)
    ret = (np.int64(1) << 31) - np.floor(rng.uniform(seed, _R_RET, i) * (1 << 30)).astype(np.int64)
    return Records(gap.astype(np.uint32), ret.astype(np.uint32), t.astype(np.uint16),
                   kv.astype(np.uint32), tier, flags.astype(np.uint8))
