"""fp64 CPU oracle for the decode-step linear layers (TEST INFRASTRUCTURE).

Only tests/, ``__graft_entry__.smoke()`` and bench.py's cpu_baseline /
reference leg may import this package.  It shares no code with the CUDA path
and never imports it.  The arithmetic lives in ``aio_oracle.c`` (plain C,
double accumulation, ascending k, OpenMP over output channels); this file
only marshals numpy arrays into it.

Functions and the passages they follow:
  * linear_bf16(x, W)        y = x W^T: the per-token weight-streaming linear
                             layer of a decode step (Sec. 2.1, Sec. 3.1).
  * linear_i8(x, q, s)       W8A16 storage-only quantization (Sec. 2.4, Sec. 6.2):
                             int8 codes dequantized with one bf16 scale per
                             output channel, exact product s*q.
  * dequant_i8(q, s)         the dequantized weights themselves.
  * bf16_to_double(h)        decoding of a bf16 bit pattern.
  * pack_tiles / unpack_tiles  the tiled weight layout the CUDA packer must
                             produce (a pure permutation; see layout.py).

Parity status: every function above is pinned by tests/test_oracle_pins.py
(brute force, one-hot, identity/zero, linearity, exact dequant, fp64 error
bound against exact rational sums) and tests/test_oracle_mutants.py.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

from .layout import ROWS_PER_GROUP, K_TILE, pack_tiles, unpack_tiles, tile_offset  # noqa: F401

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libaio_oracle.so")
_lib = None


def load(path: str = LIB_PATH):
    lib = ctypes.CDLL(path)
    i64, vp = ctypes.c_int64, ctypes.c_void_p
    lib.aio_oracle_bf16_to_double.restype = ctypes.c_double
    lib.aio_oracle_bf16_to_double.argtypes = [ctypes.c_uint16]
    lib.aio_oracle_threads.restype = ctypes.c_int
    lib.aio_oracle_threads.argtypes = []
    lib.aio_oracle_linear_bf16.restype = None
    lib.aio_oracle_linear_bf16.argtypes = [vp, vp, i64, i64, i64, vp]
    lib.aio_oracle_linear_i8.restype = None
    lib.aio_oracle_linear_i8.argtypes = [vp, vp, vp, i64, i64, i64, vp]
    lib.aio_oracle_dequant_i8.restype = None
    lib.aio_oracle_dequant_i8.argtypes = [vp, vp, i64, i64, vp]
    return lib


def _l():
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError(f"{LIB_PATH} missing: run __graft_entry__.build() first")
        _lib = load()
    return _lib


def threads() -> int:
    return int(_l().aio_oracle_threads())


def bf16_to_double(h: int) -> float:
    return float(_l().aio_oracle_bf16_to_double(int(h)))


def _c(a, dtype):
    a = np.ascontiguousarray(a)
    assert a.dtype == dtype, (a.dtype, dtype)
    return a


class Oracle:
    """Oracle bound to one compiled library (the shipped one, or a test mutant)."""

    def __init__(self, lib):
        self.lib = lib

    def linear_bf16(self, x, W):
        x = _c(x, np.uint16)
        W = _c(W, np.uint16)
        M, K = x.reshape(-1, W.shape[-1]).shape
        N = W.shape[0]
        assert W.shape == (N, K)
        y = np.empty((M, N), dtype=np.float64)
        self.lib.aio_oracle_linear_bf16(x.ctypes.data, W.ctypes.data, M, K, N, y.ctypes.data)
        return y

    def linear_i8(self, x, q, s):
        x = _c(x, np.uint16)
        q = _c(q, np.int8)
        s = _c(s, np.uint16)
        N, K = q.shape
        M = x.size // K
        assert x.size == M * K and s.shape == (N,)
        y = np.empty((M, N), dtype=np.float64)
        self.lib.aio_oracle_linear_i8(x.ctypes.data, q.ctypes.data, s.ctypes.data, M, K, N, y.ctypes.data)
        return y

    def dequant_i8(self, q, s):
        q = _c(q, np.int8)
        s = _c(s, np.uint16)
        N, K = q.shape
        Wd = np.empty((N, K), dtype=np.float64)
        self.lib.aio_oracle_dequant_i8(q.ctypes.data, s.ctypes.data, N, K, Wd.ctypes.data)
        return Wd


def _default():
    return Oracle(_l())


def linear_bf16(x, W):
    """y[m, n] = sum_k x[m, k] W[n, k] in double; x [M, K] and W [N, K] are bf16 bit patterns (uint16)."""
    return _default().linear_bf16(x, W)


def linear_i8(x, q, s):
    """y[m, n] = sum_k x[m, k] (s[n] q[n, k]) in double; q int8 [N, K], s bf16 bits [N]."""
    return _default().linear_i8(x, q, s)


def dequant_i8(q, s):
    return _default().dequant_i8(q, s)


def linear(x, W, s=None):
    """Dispatch on the weight dtype: uint16 = bf16 weights, int8 = codes with scales s."""
    if W.dtype == np.int8:
        return linear_i8(x, W, s)
    return linear_bf16(x, W)
