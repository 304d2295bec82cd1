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
