"""Parity helpers shared by the GPU tests: tolerances and oracle-side reference values.

Tolerance (per projection output [M, N], compared element by element against the fp64 oracle):
  * relative L2 error <= 1e-3 and max |err| <= 1e-2 * max |y_ref|  (the stated bar), and
  * the fp32 summation bound |y - y_ref| <= 2 (K + 1) 2^-24 sum_k |x_k w_k| + 2^-126, which any
    order of fp32 additions of exact bf16 x bf16 (or bf16 x int8) products satisfies (to first
    order (K - 1) u, doubled for margin; +1 covers the int8 scale multiply).  A dropped tile,
    a wrong row or a wrong scale breaks this bound by orders of magnitude.
"""
from __future__ import annotations

import numpy as np

import oracle

REL_L2 = 1e-3
MAX_REL = 1e-2
U32 = 2.0 ** -24


def abs_bits(h: np.ndarray) -> np.ndarray:
    return h & np.uint16(0x7FFF)


def abs_codes(q: np.ndarray):
    """|q| as int8 operands of the oracle: |q| = lo + hi with lo = min(|q|, 127) and hi = 1 exactly
    where q = -128 (|-128| = 128 does not fit int8)."""
    a = np.abs(q.astype(np.int16))
    return np.minimum(a, 127).astype(np.int8), (a == 128).astype(np.int8)


def reference(x: np.ndarray, W: np.ndarray, s=None):
    """(y_ref, sum |x_k w_k|) from the oracle; x [M, K] uint16, W [N, K] uint16 or int8."""
    if W.dtype == np.int8:
        y = oracle.linear_i8(x, W, s)
        lo, hi = abs_codes(W)
        xa = abs_bits(x)
        mag = oracle.linear_i8(xa, lo, s)
        if hi.any():
            mag = mag + oracle.linear_i8(xa, hi, s)
    else:
        y = oracle.linear_bf16(x, W)
        mag = oracle.linear_bf16(abs_bits(x), abs_bits(W))
    return y, mag


def check(y_gpu: np.ndarray, y_ref: np.ndarray, mag: np.ndarray, K: int, what: str = ""):
    y_gpu = np.asarray(y_gpu, dtype=np.float64)
    assert y_gpu.shape == y_ref.shape, (y_gpu.shape, y_ref.shape)
    assert np.all(np.isfinite(y_gpu)), f"{what}: non-finite output"
    err = np.abs(y_gpu - y_ref)
    nref = np.linalg.norm(y_ref)
    rel = np.linalg.norm(y_gpu - y_ref) / nref if nref > 0 else np.linalg.norm(y_gpu)
    assert rel <= REL_L2, f"{what}: relative L2 {rel:.3e} > {REL_L2}"
    amax = np.abs(y_ref).max()
    assert err.max() <= MAX_REL * amax + 1e-30, f"{what}: max err {err.max():.3e} > 1e-2 * {amax:.3e}"
    bound = 2.0 * (K + 1) * U32 * mag + 2.0 ** -126
    bad = err > bound
    assert not bad.any(), (f"{what}: {bad.sum()} outputs exceed the fp32 summation bound; first at "
                           f"{np.argwhere(bad)[0].tolist()}: err {err[bad][0]:.3e} bound {bound[bad][0]:.3e}")
    return rel, err.max()
