"""Reduced-precision storage of cache entries (test infrastructure, fp64 host code).

Not from the paper: an engineering variant in which the cache entries
(xhat, ehat of Eq. 3) are stored as bfloat16 while the states stay fp32. A
stored entry is the value as the GPU holds it (rounded to fp32) rounded once
more to bfloat16 -- round to nearest, ties to even, on the IEEE bit pattern:
bfloat16 keeps the sign, the 8 exponent bits and the top 7 mantissa bits of an
fp32 value.
"""
from __future__ import annotations

import numpy as np


def round_bf16(a):
    """fp64 array -> the same values rounded to fp32, then to bfloat16
    (nearest, ties to even), returned as fp64. Finite inputs only."""
    f = np.asarray(a, dtype=np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    lsb = (u >> np.uint64(16)) & np.uint64(1)          # last kept bit: ties go to even
    u = (u + np.uint64(0x7FFF) + lsb) & np.uint64(0xFFFF0000)
    return u.astype(np.uint32).view(np.float32).astype(np.float64)


STORES = {"fp32": None, "bf16": round_bf16}
