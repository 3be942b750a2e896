"""bf16 handling for the oracle (test infrastructure only).

bf16 is the upper half of an IEEE-754 binary32: 1 sign bit, 8 exponent bits, 7 stored fraction bits. The oracle
reads bf16 tensors as their uint16 bit patterns.

* ``widen``: exact. Shifting a pattern left by 16 bits gives the binary32 of the same value, and binary32 converts
  to binary64 without rounding.
* ``round_to_bf16``: binary32 -> bf16 with IEEE 754's default rounding, round to nearest with ties to even.
  Keep the top 16 bits and add one unit in their last place when the dropped 16 bits are above half an ulp, or
  exactly half with an odd kept part. NaNs stay NaN (quieted).
"""
from __future__ import annotations

import numpy as np


def widen(bits) -> np.ndarray:
    b = np.ascontiguousarray(bits, dtype=np.uint16)
    return (b.astype(np.uint32) << np.uint32(16)).view(np.float32).astype(np.float64)


def round_to_bf16(x) -> np.ndarray:
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    kept = u >> np.uint64(16)
    dropped = u & np.uint64(0xFFFF)
    half = np.uint64(0x8000)
    up = (dropped > half) | ((dropped == half) & ((kept & np.uint64(1)) == np.uint64(1)))
    r = (kept + up.astype(np.uint64)) & np.uint64(0xFFFF)
    is_nan = ((u & np.uint64(0x7F800000)) == np.uint64(0x7F800000)) & ((u & np.uint64(0x007FFFFF)) != 0)
    r = np.where(is_nan, kept | np.uint64(0x0040), r)
    return r.astype(np.uint16)
