"""Seeded synthetic inputs shared by the CUDA path and the oracle.

This module only produces input bytes (bf16 bit patterns, int8 codes); it
contains none of the linear-layer arithmetic.  The generator itself is C
(``aio_synth.c``, compiled to ``libaio_synth.so`` by ``__graft_entry__.build``)
and is counter-based, so any element of any tensor can be regenerated alone:
the oracle regenerates only the weight rows it needs for sampled checks.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB_PATH = os.path.join(_HERE, "libaio_synth.so")
_lib = None


def _load():
    global _lib
    if _lib is None:
        if not os.path.exists(_LIB_PATH):
            raise ImportError(
                f"{_LIB_PATH} is missing: run `python -c 'import __graft_entry__ as g; g.build()'` first")
        lib = ctypes.CDLL(_LIB_PATH)
        u64, dbl = ctypes.c_uint64, ctypes.c_double
        vp = ctypes.c_void_p
        lib.aio_synth_key.restype = u64
        lib.aio_synth_key.argtypes = [u64, u64, u64, u64]
        lib.aio_synth_splitmix64.restype = u64
        lib.aio_synth_splitmix64.argtypes = [u64]
        lib.aio_synth_bits.restype = u64
        lib.aio_synth_bits.argtypes = [u64, u64]
        lib.aio_synth_normal_at.restype = dbl
        lib.aio_synth_normal_at.argtypes = [u64, u64]
        lib.aio_synth_f32_to_bf16.restype = ctypes.c_uint16
        lib.aio_synth_f32_to_bf16.argtypes = [ctypes.c_float]
        lib.aio_synth_normal_bf16.restype = None
        lib.aio_synth_normal_bf16.argtypes = [u64, dbl, u64, u64, vp]
        lib.aio_synth_codes_i8.restype = None
        lib.aio_synth_codes_i8.argtypes = [u64, u64, u64, vp]
        lib.aio_synth_uniform_bf16.restype = None
        lib.aio_synth_uniform_bf16.argtypes = [u64, dbl, dbl, u64, u64, vp]
        _lib = lib
    return _lib


def key(seed: int, a: int = 0, b: int = 0, c: int = 0) -> int:
    """Stream key for one tensor: a splitmix64 chain over (seed, a, b, c)."""
    return int(_load().aio_synth_key(seed & (2**64 - 1), a, b, c))


def splitmix64(state: int) -> int:
    return int(_load().aio_synth_splitmix64(state & (2**64 - 1)))


def bits(k: int, i: int) -> int:
    return int(_load().aio_synth_bits(k, i))


def normal_at(k: int, i: int) -> float:
    return float(_load().aio_synth_normal_at(k, i))


def f32_to_bf16(f: float) -> int:
    return int(_load().aio_synth_f32_to_bf16(f))


def _dst(n, dtype, out):
    if out is None:
        arr = np.empty(n, dtype=dtype)
        return arr, arr.ctypes.data
    if isinstance(out, np.ndarray):
        assert out.dtype == dtype and out.size >= n and out.flags.c_contiguous
        return out, out.ctypes.data
    return None, int(out)  # raw host address (e.g. a pinned torch tensor)


def normal_bf16(k: int, sigma: float, n: int, offset: int = 0, out=None):
    """bf16 bit patterns of sigma * N(0,1) for elements [offset, offset + n)."""
    arr, ptr = _dst(n, np.uint16, out)
    if n:
        _load().aio_synth_normal_bf16(k, float(sigma), offset, n, ptr)
    return arr


def codes_i8(k: int, n: int, offset: int = 0, out=None):
    """int8 codes uniform on [-127, 127] for elements [offset, offset + n)."""
    arr, ptr = _dst(n, np.int8, out)
    if n:
        _load().aio_synth_codes_i8(k, offset, n, ptr)
    return arr


def uniform_bf16(k: int, lo: float, hi: float, n: int, offset: int = 0, out=None):
    """bf16 bit patterns of U(lo, hi) for elements [offset, offset + n)."""
    arr, ptr = _dst(n, np.uint16, out)
    if n:
        _load().aio_synth_uniform_bf16(k, float(lo), float(hi), offset, n, ptr)
    return arr
