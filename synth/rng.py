"""Counter-based random numbers for the synthetic workloads.

The generator is SplitMix64 (Steele, Lea and Flood, "Fast splittable
pseudorandom number generators", OOPSLA 2014): the i-th output of a stream
with state ``k`` is ``mix(k + (i + 1) * GAMMA)``, where ``mix`` is the
published 64-bit finaliser.  Because the i-th output needs no earlier one,
every draw is addressed by ``(seed, stream id, index)`` and whole arrays are
produced at once with numpy uint64 arithmetic (which wraps modulo 2**64).

Nothing here knows about sessions, scores or tiers; it only turns
addresses into uniform, normal and exponential variates.
"""
from __future__ import annotations

import numpy as np

GAMMA = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)
_S30 = np.uint64(30)
_S27 = np.uint64(27)
_S31 = np.uint64(31)
_S11 = np.uint64(11)
_INV53 = 1.0 / 9007199254740992.0  # 2**-53


def _mix(z: np.ndarray) -> np.ndarray:
    """SplitMix64 output finaliser (variant 13 of Stafford's mixers)."""
    with np.errstate(over="ignore"):
        z = (z ^ (z >> _S30)) * _M1
        z = (z ^ (z >> _S27)) * _M2
        return z ^ (z >> _S31)


def stream_key(seed: int, stream: int) -> np.uint64:
    """State word of stream ``stream`` under ``seed`` (both < 2**64)."""
    with np.errstate(over="ignore"):
        s = np.array([seed & 0xFFFFFFFFFFFFFFFF], dtype=np.uint64)
        t = np.array([(stream * 0xD1B54A32D192ED03) & 0xFFFFFFFFFFFFFFFF], dtype=np.uint64)
        return _mix(_mix(s) ^ t)[0]


def u64(seed: int, stream: int, index) -> np.ndarray:
    """Raw 64-bit outputs at the given indices of one stream."""
    idx = np.asarray(index, dtype=np.uint64)
    k = stream_key(seed, stream)
    with np.errstate(over="ignore"):
        return _mix(k + (idx + np.uint64(1)) * GAMMA)


def uniform_open0(seed: int, stream: int, index) -> np.ndarray:
    """Uniform doubles in (0, 1]: 53 random bits, shifted up by one ulp."""
    x = u64(seed, stream, index)
    return ((x >> _S11).astype(np.float64) + 1.0) * _INV53


def uniform(seed: int, stream: int, index) -> np.ndarray:
    """Uniform doubles in [0, 1)."""
    x = u64(seed, stream, index)
    return (x >> _S11).astype(np.float64) * _INV53


def randint(seed: int, stream: int, index, lo: int, hi: int) -> np.ndarray:
    """Uniform integers in the closed range [lo, hi]."""
    u = uniform(seed, stream, index)
    v = lo + np.floor(u * (hi - lo + 1)).astype(np.int64)
    return np.minimum(v, hi)


def normal(seed: int, stream: int, index) -> np.ndarray:
    """Standard normals by the Box-Muller transform (Box and Muller, 1958).

    Stream ``stream`` supplies the radius draw and ``stream + 1`` the angle.
    """
    u1 = uniform_open0(seed, stream, index)
    u2 = uniform(seed, stream + 1, index)
    return np.sqrt(-2.0 * np.log(u1)) * np.cos(2.0 * np.pi * u2)


def exponential(seed: int, stream: int, index, mean: float) -> np.ndarray:
    """Exponential variates with the given mean, by inversion."""
    return -np.log(uniform_open0(seed, stream, index)) * mean
