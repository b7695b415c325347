"""Plant mistakes in the oracle (CPU only) and check that the pins catch each one.

Each mutant is the oracle C source compiled with AIO_ORACLE_MUTANT=k:
  1 dropped term, 2 transposed operand, 3 wrong sign, 4 wrong scale index,
  5 dequantized weight rounded to bf16 before the product, 6 lost code sign,
  7 bf16 rounding toward zero, 8 sign error in the logistic of silu,
  9 RMSNorm mean over K - 1, 10 SwiGLU gate and up swapped,
  11 attention without the 1/sqrt(d) scale, 12 causal limit off by one, 13 attention output not
  normalised.
"""
import math
import struct
from fractions import Fraction

import numpy as np
import pytest

import oracle
import synth
from oracle import build as ob


def _bf16_int(v):
    return struct.unpack("<I", struct.pack("<f", float(v)))[0] >> 16


def _exact(h):
    h = int(h)
    sign = -1 if h & 0x8000 else 1
    e, m = (h >> 7) & 0xFF, h & 0x7F
    return sign * (1 + Fraction(m, 128)) * Fraction(2) ** (e - 127) if e else sign * Fraction(m, 128) * Fraction(2) ** -126


def pins_hold(o: oracle.Oracle) -> bool:
    rng = np.random.default_rng(0)
    # brute force, integer-valued bf16
    xi = rng.integers(-8, 9, size=(2, 12))
    wi = rng.integers(-8, 9, size=(5, 12))
    to = np.vectorize(_bf16_int, otypes=[np.uint16])
    y = o.linear_bf16(to(xi), to(wi))
    if not np.array_equal(y, xi @ wi.T):
        return False
    # one-hot column selection with N != K
    K, N = 9, 4
    W = synth.normal_bf16(synth.key(1), 1.0, N * K).reshape(N, K)
    for k in range(K):
        x = np.zeros((1, K), np.uint16)
        x[0, k] = _bf16_int(1)
        if [Fraction(v) for v in o.linear_bf16(x, W)[0]] != [_exact(W[n, k]) for n in range(N)]:
            return False
    # int8: one-hot with distinct scales, and exact dequant of known codes
    q = rng.integers(-127, 128, size=(N, K)).astype(np.int8)
    s = synth.uniform_bf16(synth.key(2), 1e-3, 1e-2, N)
    for k in range(K):
        x = np.zeros((1, K), np.uint16)
        x[0, k] = _bf16_int(1)
        y = o.linear_i8(x, q, s)
        if any(Fraction(y[0, n]) != _exact(s[n]) * int(q[n, k]) for n in range(N)):
            return False
    x = np.array([[_bf16_int(1)]], np.uint16)
    if o.linear_i8(x, np.array([[127]], np.int8), np.array([0x3BA4], np.uint16))[0, 0] != 0.6356201171875:
        return False
    return True


def chain_pins_hold(o: oracle.Oracle) -> bool:
    """A few of tests/test_oracle_chain_pins.py's facts, evaluated on an arbitrary build."""
    if o.double_to_bf16(1 + 3 * 2 ** -8) != 0x3F82 or o.double_to_bf16(1 + 2 ** -8 + 2 ** -30) != 0x3F81:
        return False
    if abs(o.silu(math.log(3)) - 0.75 * math.log(3)) > 1e-15:
        return False
    g = np.array([_bf16_int(v) for v in (1.0, 1.0, 0.5, 2.0)], np.uint16)
    _, x = o.rmsnorm(np.array([[3.0, 4.0, 0.0, 0.0]], np.float32), None, g, 39 / 4)   # rms 4
    if [int(v) for v in x[0]] != [0x3F40, 0x3F80, 0, 0]:
        return False
    t = float(np.float32(math.log(3)))
    y = np.array([[t, 0.0, np.float32(4 / (3 * t)), 2.0]], np.float32)             # gate | up, I = 2
    if [int(v) for v in o.swiglu(y, 2)[0]] != [0x3F80, 0]:
        return False
    return True


def attention_pins_hold(o: oracle.Oracle) -> bool:
    """A few of tests/test_oracle_attention_pins.py's facts, evaluated on an arbitrary build."""
    d, L = 16, 2
    k = np.zeros((1, L, d), np.uint16)
    k[0, 0, 0] = _bf16_int(1)
    v = np.zeros((1, L, d), np.uint16)
    v[0, 0, 0] = _bf16_int(1)
    v[0, 1, 1] = _bf16_int(1)
    q = np.zeros((1, d), np.float32)
    q[0, 0] = np.float32(math.sqrt(d) * math.log(3))
    out = o.attention(q, k, v, L)
    w0 = 1 / (1 + math.exp(-float(q[0, 0]) / math.sqrt(d)))
    if abs(out[0, 0] - w0) > 1e-15 or abs(out[0, 1] - (1 - w0)) > 1e-15:
        return False
    L, M = 4, 2
    k = np.zeros((1, L, 4), np.uint16)
    for j in range(L):
        k[0, j, 0] = _bf16_int(j)
    v = np.zeros((1, L, 4), np.uint16)
    for j in range(L):
        v[0, j, 0] = _bf16_int(j + 1)
    q = np.zeros((M, 4), np.float32)
    q[:, 0] = 1e5
    out = o.attention(q, k, v, L)
    return out[0, 0] == 3.0 and out[1, 0] == 4.0


def test_shipped_oracle_passes_pins():
    o = oracle.Oracle(oracle.load())
    assert pins_hold(o) and chain_pins_hold(o) and attention_pins_hold(o)


@pytest.mark.parametrize("mutant", [1, 2, 3, 4, 5, 6])
def test_mutant_is_caught(tmp_path, mutant):
    path = ob.build(out=str(tmp_path / f"libaio_oracle_m{mutant}.so"), mutant=mutant)
    assert not pins_hold(oracle.Oracle(oracle.load(path)))


@pytest.mark.parametrize("mutant", [7, 8, 9, 10])
def test_chain_mutant_is_caught(tmp_path, mutant):
    path = ob.build(out=str(tmp_path / f"libaio_oracle_m{mutant}.so"), mutant=mutant)
    assert not chain_pins_hold(oracle.Oracle(oracle.load(path)))


@pytest.mark.parametrize("mutant", [11, 12, 13])
def test_attention_mutant_is_caught(tmp_path, mutant):
    path = ob.build(out=str(tmp_path / f"libaio_oracle_m{mutant}.so"), mutant=mutant)
    assert not attention_pins_hold(oracle.Oracle(oracle.load(path)))
