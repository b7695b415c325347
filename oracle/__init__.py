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
  * double_to_bf16(v)        round a double to bf16, nearest-even.
  * attention(q, k, v, L)    decode attention of M new tokens over a KV cache of
                             L positions (the long-context path, Sec. 3.3, Sec. 5.1).
  * pld.draft / pld.argmax / pld.accept  prompt-lookup drafting (N = 6, L = 2,
                             Sec. 4.2) and greedy acceptance of the verification
                             pass (oracle/pld.py, plain Python).
  * attention_link(y_qkv, kv, L_past, n_heads)
                             the chained step's attention between QKV and O:
                             the new tokens' k and v appended to the layer's KV
                             cache, decode attention over it, x = bf16(out)
                             (Sec. 3.3, Sec. 5.1: 2K and 32K contexts).
  * silu(t), rmsnorm(...), swiglu(...), slice_x(...)
                             the steps between the projections of a chained
                             decoder step; chain_step(...) runs a whole chained
                             step.  The paper prints no block structure (it
                             names its models, Sec. 4.2): the reading is a
                             pre-norm decoder block (RMSNorm, attention, SwiGLU
                             MLP, residual adds) whose attention covers one
                             position, so it returns the V third of QKV.

Parity status: every function above is pinned by tests/test_oracle_pins.py
(brute force, one-hot, identity/zero, linearity, exact dequant, fp64 error
bound against exact rational sums), tests/test_oracle_chain_pins.py (bf16
rounding against exact rationals and a library conversion, closed forms of the
logistic, RMSNorm invariants, exact residual adds),
tests/test_oracle_attention_pins.py, tests/test_oracle_pld_pins.py and
tests/test_oracle_mutants.py.
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
    lib.aio_oracle_double_to_bf16.restype = ctypes.c_uint16
    lib.aio_oracle_double_to_bf16.argtypes = [ctypes.c_double]
    lib.aio_oracle_silu.restype = ctypes.c_double
    lib.aio_oracle_silu.argtypes = [ctypes.c_double]
    lib.aio_oracle_rmsnorm.restype = None
    lib.aio_oracle_rmsnorm.argtypes = [vp, vp, vp, i64, i64, ctypes.c_double, vp, vp]
    lib.aio_oracle_swiglu.restype = None
    lib.aio_oracle_swiglu.argtypes = [vp, i64, i64, i64, vp]
    lib.aio_oracle_slice.restype = None
    lib.aio_oracle_slice.argtypes = [vp, i64, i64, i64, i64, vp]
    lib.aio_oracle_attention.restype = None
    lib.aio_oracle_attention.argtypes = [vp, i64, vp, vp, i64, i64, i64, i64, i64, vp]
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

    def double_to_bf16(self, v) -> int:
        return int(self.lib.aio_oracle_double_to_bf16(float(v)))

    def silu(self, t) -> float:
        return float(self.lib.aio_oracle_silu(float(t)))

    def rmsnorm(self, h_in, r, gamma, eps):
        """(h_out, x): h_out = fp32(h_in + r) (r may be None), x = bf16(h_out * gamma / rms(h_out))."""
        h_in = _c(h_in, np.float32)
        M, K = h_in.shape
        rr = None if r is None else _c(r, np.float32).reshape(M, K)
        g = _c(gamma, np.uint16)
        assert g.shape == (K,)
        h_out = np.empty((M, K), np.float32)
        x = np.empty((M, K), np.uint16)
        self.lib.aio_oracle_rmsnorm(h_in.ctypes.data, None if rr is None else rr.ctypes.data, g.ctypes.data, M, K,
                                    float(eps), h_out.ctypes.data, x.ctypes.data)
        return h_out, x

    def swiglu(self, y, I):
        """x[m, k] = bf16(silu(y[m, k]) * y[m, I + k]) for k < I; y [M, stride >= 2I] fp32."""
        y = _c(y, np.float32)
        M, stride = y.shape
        assert stride >= 2 * I
        x = np.empty((M, I), np.uint16)
        self.lib.aio_oracle_swiglu(y.ctypes.data, M, I, stride, x.ctypes.data)
        return x

    def slice_x(self, y, off, K):
        """x[m, k] = bf16(y[m, off + k]) for k < K."""
        y = _c(y, np.float32)
        M, stride = y.shape
        assert 0 <= off and off + K <= stride
        x = np.empty((M, K), np.uint16)
        self.lib.aio_oracle_slice(y.ctypes.data, M, K, stride, off, x.ctypes.data)
        return x

    def attention(self, q, k, v, L, M=None):
        """Decode attention: q [M, n_heads d] fp32 (rows may be wider: only the first n_heads d
        columns are read), k, v [n_heads, L_max, d] bf16 bits; the M new tokens sit at positions
        L - M .. L - 1 and attend causally.  Returns out [M, n_heads d] in double."""
        q = _c(q, np.float32)
        k = _c(k, np.uint16)
        v = _c(v, np.uint16)
        n_heads, L_max, d = k.shape
        M = q.shape[0] if M is None else M
        assert v.shape == k.shape and 1 <= L <= L_max and M <= L and q.shape[1] >= n_heads * d
        out = np.empty((M, n_heads * d), np.float64)
        self.lib.aio_oracle_attention(q.ctypes.data, q.shape[1], k.ctypes.data, v.ctypes.data, n_heads, d, L_max, L, M,
                                      out.ctypes.data)
        return out

    def round_bf16(self, v):
        """Each double of v rounded to bf16 (nearest, ties to even), as bf16 bits."""
        v = np.asarray(v, dtype=np.float64)
        return np.array([self.double_to_bf16(t) for t in v.ravel()], dtype=np.uint16).reshape(v.shape)

    def attention_link(self, y_qkv, kv, L_past, n_heads, d=128):
        """x of O when the new tokens attend over a KV cache (the chained step's attention link).
        y_qkv [M, >= 3 n_heads d] fp32 is the QKV output: q, k, v are its column thirds, head h at
        columns [h d, h d + d) of each.  kv [2, n_heads, L_max, d] bf16 bits is the layer's cache (K
        then V) holding L_past positions.  Steps: the new tokens' k and v, rounded to bf16, are
        written at positions L_past .. L_past + M - 1; token m attends to positions
        j <= L_past + m (decode attention over L = L_past + M positions); x = bf16(out).
        Returns (x [M, n_heads d] bf16 bits, the updated cache)."""
        y = np.ascontiguousarray(y_qkv, dtype=np.float32)
        M = y.shape[0]
        H = n_heads * d
        kv = np.array(kv, dtype=np.uint16, copy=True)
        assert kv.shape[:2] == (2, n_heads) and kv.shape[3] == d and L_past + M <= kv.shape[2]
        k_new = self.slice_x(y, H, H).reshape(M, n_heads, d)
        v_new = self.slice_x(y, 2 * H, H).reshape(M, n_heads, d)
        kv[0, :, L_past:L_past + M, :] = k_new.transpose(1, 0, 2)
        kv[1, :, L_past:L_past + M, :] = v_new.transpose(1, 0, 2)
        out = self.attention(y, kv[0], kv[1], L_past + M, M)
        return self.round_bf16(out), kv

    def prep(self, link, ys, h, h0, gammas, eps, caches=None):
        """x of one projection of a chained step from the buffers before it (``link``: a
        synth.workloads.ChainLink); returns (x, h_out or None).  ys: fp32 y of earlier projections
        by index; h: the two residual buffers; h0: the step's input residual stream; caches: for
        attention links, a dict layer -> [kv, L_past, n_heads] whose kv the link replaces with the
        updated cache."""
        from synth.workloads import XOP_RMSNORM, XOP_SWIGLU, XOP_SLICE, XOP_ATTENTION
        if link.op == XOP_ATTENTION:
            c = caches[link.layer]
            x, c[0] = self.attention_link(ys[link.src], c[0], c[1], c[2])
            return x, None
        if link.op == XOP_RMSNORM:
            h_in = h0 if link.h_in < 0 else h[link.h_in]
            r = None if link.src < 0 else ys[link.src]
            h_out, x = self.rmsnorm(h_in, r, gammas[link.gamma], eps)
            return x, (h_out if link.h_out >= 0 else None)
        if link.op == XOP_SWIGLU:
            y = ys[link.src]
            return self.swiglu(y, y.shape[1] // 2), None
        if link.op == XOP_SLICE:
            return self.slice_x(ys[link.src], link.src_off, link.K), None
        raise ValueError(link.op)

    def chain_step(self, links, weights, h0, gammas, eps, caches=None):
        """A whole chained decoder step in the oracle's own arithmetic: every projection's x from
        the oracle's earlier outputs, y rounded to fp32 as the CUDA path stores it.  weights[i] is
        W (bf16 bits) or (q, s) for int8; caches as for prep (updated in place).  Returns
        (xs, ys, h) with ys in fp32."""
        xs, ys = [], []
        h = [None, None]
        for link, w in zip(links, weights):
            x, h_out = self.prep(link, ys, h, h0, gammas, eps, caches)
            if h_out is not None:
                h[link.h_out] = h_out
            y = self.linear_i8(x, *w) if isinstance(w, tuple) else self.linear_bf16(x, w)
            xs.append(x)
            ys.append(y.astype(np.float32))
        return xs, ys, h


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


def double_to_bf16(v) -> int:
    return _default().double_to_bf16(v)


def silu(t) -> float:
    return _default().silu(t)


def rmsnorm(h_in, r, gamma, eps):
    return _default().rmsnorm(h_in, r, gamma, eps)


def swiglu(y, I):
    return _default().swiglu(y, I)


def slice_x(y, off, K):
    return _default().slice_x(y, off, K)


def chain_step(links, weights, h0, gammas, eps, caches=None):
    return _default().chain_step(links, weights, h0, gammas, eps, caches)


def attention_link(y_qkv, kv, L_past, n_heads, d=128):
    return _default().attention_link(y_qkv, kv, L_past, n_heads, d)


def attention(q, k, v, L, M=None):
    return _default().attention(q, k, v, L, M)
