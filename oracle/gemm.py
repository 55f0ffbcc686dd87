"""fp64 reference GEMM over bf16 inputs — TEST INFRASTRUCTURE ONLY.

Definition followed (Sec. 2.1.2): C (M x N) is the product of A (M x K) and
B, with 2*M*N*K multiplies and adds.  The workloads store A as M x K row-major
and B as K x N row-major, both bf16, so ``ref[i, j] = sum_k A[i, k] * B[k, j]``.
The sum runs in increasing k in double precision (``oracle_gemm.c``); inputs
arrive as raw uint16 bf16 bit patterns so both sides read identical bits.

``gemm_python`` is the same definition as a pure-Python triple loop, for tiny
shapes only; it exists to pin the C implementation.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

from . import build as _build

_lib = None


def _load():
    global _lib
    if _lib is None:
        path = _build.build()
        lib = ctypes.CDLL(path)
        i64, p = ctypes.c_int64, ctypes.c_void_p
        lib.oracle_gemm_bf16.argtypes = [p, i64, p, i64, p, i64, i64, i64, i64]
        lib.oracle_gemm_bf16.restype = None
        lib.oracle_gemm_bf16_rows.argtypes = [p, i64, p, i64, p, i64, p, i64, i64]
        lib.oracle_gemm_bf16_rows.restype = None
        lib.oracle_gemm_bf16_entries.argtypes = [p, i64, p, i64, p, p, i64, p, i64]
        lib.oracle_gemm_bf16_entries.restype = None
        lib.oracle_bf16_decode.argtypes = [p, p, i64]
        lib.oracle_bf16_decode.restype = None
        lib.oracle_num_threads.argtypes = []
        lib.oracle_num_threads.restype = ctypes.c_int
        lib.oracle_set_threads.argtypes = [ctypes.c_int]
        lib.oracle_set_threads.restype = None
        _lib = lib
    return _lib


def _as_bits(x: np.ndarray) -> np.ndarray:
    x = np.ascontiguousarray(x)
    if x.dtype != np.uint16:
        raise TypeError("oracle inputs are raw bf16 bit patterns (uint16)")
    return x


def num_threads() -> int:
    """Threads the C oracle's OpenMP loops use."""
    return int(_load().oracle_num_threads())


def set_threads(n: int) -> None:
    _load().oracle_set_threads(int(n))


def bf16_decode(bits: np.ndarray) -> np.ndarray:
    """Exact value (float64) of each bf16 bit pattern, via the C decoder."""
    bits = _as_bits(bits)
    out = np.empty(bits.shape, dtype=np.float64)
    _load().oracle_bf16_decode(bits.ctypes.data, out.ctypes.data, bits.size)
    return out


def gemm(a_bits: np.ndarray, b_bits: np.ndarray) -> np.ndarray:
    """ref = A @ B in fp64 for A (M x K) and B (K x N) given as bf16 bits."""
    a = _as_bits(a_bits)
    b = _as_bits(b_bits)
    if a.ndim != 2 or b.ndim != 2 or a.shape[1] != b.shape[0]:
        raise ValueError(f"shape mismatch {a.shape} x {b.shape}")
    M, K = a.shape
    N = b.shape[1]
    out = np.empty((M, N), dtype=np.float64)
    if M and N:
        _load().oracle_gemm_bf16(a.ctypes.data, K, b.ctypes.data, N,
                                 out.ctypes.data, N, M, N, K)
    return out


def gemm_rows(a_bits: np.ndarray, b_bits: np.ndarray, rows) -> np.ndarray:
    """Rows ``rows`` of A @ B (fp64), each computed exactly as in ``gemm``."""
    a = _as_bits(a_bits)
    b = _as_bits(b_bits)
    M, K = a.shape
    N = b.shape[1]
    rows = np.ascontiguousarray(np.asarray(rows, dtype=np.int64))
    if rows.size and (rows.min() < 0 or rows.max() >= M):
        raise IndexError("row index out of range")
    out = np.empty((rows.size, N), dtype=np.float64)
    if rows.size and N:
        _load().oracle_gemm_bf16_rows(a.ctypes.data, K, b.ctypes.data, N,
                                      rows.ctypes.data, rows.size, out.ctypes.data, N, K)
    return out


def gemm_entries(a_bits: np.ndarray, b_bits: np.ndarray, ii, jj) -> np.ndarray:
    """Entries (ii[t], jj[t]) of A @ B in fp64."""
    a = _as_bits(a_bits)
    b = _as_bits(b_bits)
    M, K = a.shape
    N = b.shape[1]
    ii = np.ascontiguousarray(np.asarray(ii, dtype=np.int64))
    jj = np.ascontiguousarray(np.asarray(jj, dtype=np.int64))
    if ii.shape != jj.shape:
        raise ValueError("ii and jj differ in length")
    if ii.size and (ii.min() < 0 or ii.max() >= M or jj.min() < 0 or jj.max() >= N):
        raise IndexError("entry index out of range")
    out = np.empty(ii.size, dtype=np.float64)
    if ii.size:
        _load().oracle_gemm_bf16_entries(a.ctypes.data, K, b.ctypes.data, N,
                                         ii.ctypes.data, jj.ctypes.data, ii.size,
                                         out.ctypes.data, K)
    return out


def _bf16_value_python(h: int) -> float:
    """Value of one bf16 bit pattern from the format's fields (sign, 8-bit
    biased exponent, 7-bit fraction), written out independently of the C
    decoder's bit shift."""
    sign = -1.0 if (h >> 15) & 1 else 1.0
    e = (h >> 7) & 0xFF
    f = h & 0x7F
    if e == 0xFF:
        return sign * float("inf") if f == 0 else float("nan")
    if e == 0:
        return sign * (f / 128.0) * 2.0 ** (-126)
    return sign * (1.0 + f / 128.0) * 2.0 ** (e - 127)


def gemm_python(a_bits, b_bits):
    """Pure-Python triple loop of the same definition (tiny shapes only)."""
    a = [[_bf16_value_python(int(v)) for v in row] for row in np.asarray(a_bits)]
    b = [[_bf16_value_python(int(v)) for v in row] for row in np.asarray(b_bits)]
    M = len(a)
    K = len(b)
    N = len(b[0]) if K else 0
    out = [[0.0] * N for _ in range(M)]
    for i in range(M):
        for j in range(N):
            s = 0.0
            for k in range(K):
                s += a[i][k] * b[k][j]
            out[i][j] = s
    return np.array(out, dtype=np.float64).reshape(M, N)


def bf16_value_python(h: int) -> float:
    return _bf16_value_python(h)


def tolerance(ref: np.ndarray) -> float:
    """Per-GEMM acceptance bound |gpu - ref| <= 1e-2 * max|ref| + 1e-3 for
    bf16 inputs with fp32 accumulation (the bar the hot path is held to)."""
    m = float(np.max(np.abs(ref))) if ref.size else 0.0
    return 1e-2 * m + 1e-3


__all__ = ["gemm", "gemm_rows", "gemm_entries", "gemm_python", "bf16_decode",
           "bf16_value_python", "tolerance", "num_threads", "set_threads"]

if os.environ.get("GOLDY_ORACLE_THREADS"):
    set_threads(int(os.environ["GOLDY_ORACLE_THREADS"]))


def gemm_batched(a_bits: np.ndarray, b_bits: np.ndarray) -> np.ndarray:
    """A strided batch of GEMMs (Sec. 6.7's B-GEMMs): entry i of the result
    is gemm(a_bits[i], b_bits[i]) for a_bits (batch x M x K) and b_bits
    (batch x K x N)."""
    a_bits = _as_bits(a_bits)
    b_bits = _as_bits(b_bits)
    if a_bits.ndim != 3 or b_bits.ndim != 3 or a_bits.shape[0] != b_bits.shape[0]:
        raise ValueError("batched operands must be (batch, rows, cols) with equal batch")
    out = np.empty((a_bits.shape[0], a_bits.shape[1], b_bits.shape[2]), dtype=np.float64)
    for i in range(a_bits.shape[0]):
        out[i] = gemm(a_bits[i], b_bits[i])
    return out
