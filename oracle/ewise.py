"""Element-wise add Z = X + Y — TEST INFRASTRUCTURE ONLY.

The non-GEMM kernel the paper co-schedules with a GEMM (Sec. 7.1).  The
operation is defined at the precision the kernel computes in (the paper
fixes none): each bf16 input is widened exactly to fp32, the two are added
with one IEEE-754 binary32 addition (round to nearest, ties to even), and for
bf16 output the fp32 sum is rounded to bf16 to nearest, ties to even.  numpy's
float32 addition is that IEEE operation; the bf16 rounding is written out
here on the bit pattern.
"""
from __future__ import annotations

import numpy as np


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    """Exact widening: a bf16 pattern is the top half of the binary32 one."""
    return (bits.astype(np.uint32) << 16).view(np.float32)


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round binary32 values to bf16 patterns, to nearest, ties to even:
    add 0x7FFF plus the lowest kept bit to the pattern and truncate.  NaNs
    keep a quiet NaN pattern (they do not occur in the tests' inputs)."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    keep = (u >> 16) & 1
    r = ((u + 0x7FFF + keep) >> 16).astype(np.uint16)
    nan = np.isnan(x)
    if nan.any():
        r[nan] = ((u[nan] >> 16) | 0x40).astype(np.uint16)
    return r


def add_bf16(x_bits: np.ndarray, y_bits: np.ndarray) -> np.ndarray:
    """bf16 patterns of X + Y."""
    s = bf16_bits_to_f32(x_bits) + bf16_bits_to_f32(y_bits)     # one binary32 addition, RNE
    return f32_to_bf16_bits(s)


def add_f32(x: np.ndarray, y: np.ndarray) -> np.ndarray:
    return np.asarray(x, dtype=np.float32) + np.asarray(y, dtype=np.float32)
