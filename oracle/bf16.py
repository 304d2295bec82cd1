"""Exact widening of bf16 bit patterns to float64 (oracle side).

A bf16 value is the top 16 bits of an IEEE-754 binary32; shifting the pattern
left by 16 gives that binary32 exactly, and binary32 -> binary64 is exact.
"""
import numpy as np


def widen(bits: np.ndarray) -> np.ndarray:
    bits = np.asarray(bits)
    if bits.dtype == np.float32 or bits.dtype == np.float64:
        return bits.astype(np.float64)
    assert bits.dtype == np.uint16, bits.dtype
    return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def round_to_bf16(x: np.ndarray) -> np.ndarray:
    """Nearest bf16 value of each float64 (ties to even), returned as float64.

    bf16 keeps 8 significant bits: write x = m * 2^e with m in [0.5, 1), round
    m * 2^8 to the nearest integer (half to even) and scale back.  Values here
    are normal and far from the bf16 range limits.
    """
    x = np.asarray(x, np.float64)
    m, e = np.frexp(x)
    return np.ldexp(np.round(np.ldexp(m, 8)), e - 8)
