"""Counter-based SplitMix64 streams and Box-Muller normals (numpy, vectorised).

SplitMix64 is the generator of Steele, Lea and Flood, "Fast splittable
pseudorandom number generators" (OOPSLA 2014), in the form Vigna publishes
as the seeding generator of the xoshiro family: the state advances by the
golden-ratio increment 0x9E3779B97F4A7C15 and each output is the state passed
through a fixed 64-bit finaliser.  Because the state after i steps is simply
``seed + i * gamma``, output i can be computed directly, so a whole array is
one vectorised expression and any element can be regenerated on its own.

Normals use the Box-Muller transform (Box and Muller, 1958): two independent
uniforms u1 in (0, 1] and u2 in [0, 1) give sqrt(-2 ln u1) * cos(2 pi u2).

This module only draws random numbers for synthetic inputs.  It contains none
of the scoring arithmetic and is shared by the CUDA-path tests, the oracle and
the benchmark alike.
"""
from __future__ import annotations

import numpy as np

_GAMMA = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)
_MASK64 = (1 << 64) - 1


def _mix(z: np.ndarray) -> np.ndarray:
    """SplitMix64 output finaliser on a uint64 array (wrapping arithmetic)."""
    z = z.copy()
    z ^= z >> np.uint64(30)
    z *= _M1
    z ^= z >> np.uint64(27)
    z *= _M2
    z ^= z >> np.uint64(31)
    return z


def _mix_scalar(z: int) -> int:
    z &= _MASK64
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & _MASK64
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & _MASK64
    return z ^ (z >> 31)


def _fnv1a64(text: str) -> int:
    h = 0xCBF29CE484222325
    for byte in text.encode("utf-8"):
        h ^= byte
        h = (h * 0x100000001B3) & _MASK64
    return h


def stream_seed(seed: int, tag: str) -> int:
    """Seed of the named sub-stream ``tag`` of master seed ``seed``."""
    return _mix_scalar(_mix_scalar(seed & _MASK64) ^ _fnv1a64(tag))


class Stream:
    """One SplitMix64 stream; successive draws continue where the last ended."""

    def __init__(self, seed: int, tag: str):
        self.state = stream_seed(seed, tag)
        self.count = 0

    def u64(self, n: int) -> np.ndarray:
        with np.errstate(over="ignore"):
            i = np.arange(self.count + 1, self.count + 1 + n, dtype=np.uint64)
            z = np.uint64(self.state) + i * _GAMMA
            out = _mix(z)
        self.count += n
        return out

    def uniform(self, n: int) -> np.ndarray:
        """Doubles in [0, 1) with 53 random bits."""
        return (self.u64(n) >> np.uint64(11)).astype(np.float64) * (1.0 / 9007199254740992.0)

    def normal(self, n: int) -> np.ndarray:
        """Standard normals by Box-Muller (one normal per uniform pair)."""
        u1 = 1.0 - self.uniform(n)  # (0, 1]
        u2 = self.uniform(n)
        return np.sqrt(-2.0 * np.log(u1)) * np.cos(2.0 * np.pi * u2)

    def integers(self, lo: int, hi: int, n: int) -> np.ndarray:
        """Integers uniform on [lo, hi] inclusive (hi - lo < 2**31)."""
        span = hi - lo + 1
        v = np.floor(self.uniform(n) * span).astype(np.int64)
        return np.minimum(v, span - 1) + lo
