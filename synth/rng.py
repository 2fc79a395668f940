"""Counter-based random numbers and bf16 bit handling for the input generators.

``splitmix64`` is the finaliser of Steele, Lea and Flood's SplitMix generator with the constants
Vigna published for ``splitmix64`` (public domain).  The harness draws every random number from
``harness_key(seed, row, step, slot)``, a fixed chain of splitmix64 calls, so the host and the device
produce identical streams without sharing state.
"""
from __future__ import annotations

import numpy as np

_GOLDEN = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)
_MASK = (1 << 64) - 1


def splitmix64(z):
    """Vectorised splitmix64 on uint64 arrays (wrapping arithmetic)."""
    z = np.asarray(z, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = z + _GOLDEN
        z = (z ^ (z >> np.uint64(30))) * _M1
        z = (z ^ (z >> np.uint64(27))) * _M2
    return z ^ (z >> np.uint64(31))


def splitmix64_int(z: int) -> int:
    """Scalar splitmix64 on Python ints (used to pin the vectorised version)."""
    z = (z + 0x9E3779B97F4A7C15) & _MASK
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & _MASK
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & _MASK
    return z ^ (z >> 31)


def harness_key(seed, row, step, slot):
    """Random word for (seed, row, step, slot): splitmix64 applied along the chain
    seed -> row -> step -> slot, each stage xor-ing the next coordinate in."""
    k = splitmix64(np.uint64(seed))
    k = splitmix64(k ^ np.asarray(row, dtype=np.uint64))
    k = splitmix64(k ^ np.asarray(step, dtype=np.uint64))
    return splitmix64(k ^ np.asarray(slot, dtype=np.uint64))


def bf16_bits_from_f32(f) -> np.ndarray:
    """Round binary32 values to bf16 (round to nearest, ties to even); returns the uint16 bits."""
    f = np.ascontiguousarray(f, dtype=np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    r = (u + np.uint64(0x7FFF) + ((u >> np.uint64(16)) & np.uint64(1))) >> np.uint64(16)
    return r.astype(np.uint16)


def f32_from_bf16_bits(bits) -> np.ndarray:
    b = np.ascontiguousarray(bits, dtype=np.uint16)
    return (b.astype(np.uint32) << np.uint32(16)).view(np.float32)
