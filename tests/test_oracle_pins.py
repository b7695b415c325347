"""Pins for the fp64 oracle: facts fixed by the mathematics, not by the oracle itself (CPU).

The paper prints no worked numeric example of a linear layer, so the oracle is
pinned by closed forms and invariants of y = x W^T (the per-token weight
streaming of Sec. 2.1 / Sec. 3.1) and of W8A16 dequantization (Sec. 2.4):
brute force against exact integer sums, one-hot inputs selecting one weight
column, identity and zero weights, linearity and homogeneity, exact dequant
of known codes, and the fp64 error bound against exact rational sums.
Each check is written so that a dropped term, a wrong sign, a wrong index,
a transposed operand or a rounded dequant fails it (see test_oracle_mutants).
"""
import os
import struct
from fractions import Fraction

import numpy as np
import pytest

import oracle
import synth
from synth import workloads as wl


def bf16_of_int(v):
    """bf16 bit pattern of a small integer (exact for |v| <= 256)."""
    assert abs(v) <= 256
    b = struct.unpack("<I", struct.pack("<f", float(v)))[0]
    assert b & 0xFFFF == 0
    return b >> 16


def bf16_value_exact(h):
    """Exact rational value of a finite bf16 bit pattern (sign, exponent, mantissa)."""
    h = int(h)
    sign = -1 if h & 0x8000 else 1
    e = (h >> 7) & 0xFF
    m = h & 0x7F
    assert e != 0xFF
    if e == 0:
        return sign * Fraction(m, 128) * Fraction(2) ** (-126)
    return sign * (1 + Fraction(m, 128)) * Fraction(2) ** (e - 127)


def rand_int_bf16(rng, shape, lo=-8, hi=8):
    ints = rng.integers(lo, hi + 1, size=shape)
    return ints, np.vectorize(bf16_of_int, otypes=[np.uint16])(ints)


# ---------------------------------------------------------------- brute force
@pytest.mark.parametrize("M,K,N", [(1, 1, 1), (1, 5, 3), (2, 16, 8), (3, 32, 7), (3, 17, 5)])
def test_bruteforce_integer_bf16(M, K, N):
    rng = np.random.default_rng(M * 100 + K * 10 + N)
    xi, x = rand_int_bf16(rng, (M, K))
    wi, W = rand_int_bf16(rng, (N, K))
    y = oracle.linear_bf16(x, W)
    for m in range(M):
        for n in range(N):
            exact = sum(int(xi[m, k]) * int(wi[n, k]) for k in range(K))
            assert y[m, n] == exact


@pytest.mark.parametrize("M,K,N", [(1, 16, 4), (2, 32, 8), (3, 48, 3)])
def test_bruteforce_integer_i8(M, K, N):
    rng = np.random.default_rng(K + N)
    xi, x = rand_int_bf16(rng, (M, K))
    q = rng.integers(-127, 128, size=(N, K)).astype(np.int8)
    si = rng.integers(1, 9, size=N)
    s = np.vectorize(bf16_of_int, otypes=[np.uint16])(si)
    y = oracle.linear_i8(x, q, s)
    for m in range(M):
        for n in range(N):
            exact = int(si[n]) * sum(int(xi[m, k]) * int(q[n, k]) for k in range(K))
            assert y[m, n] == exact


# ---------------------------------------------------------------- one-hot / identity / zero
def test_one_hot_selects_weight_column_bf16():
    K, N = 24, 10   # N != K so a transposed read cannot pass
    k_ = synth.key(11)
    W = synth.normal_bf16(k_, 1.0, N * K).reshape(N, K)
    one = bf16_of_int(1)
    for k in range(K):
        x = np.zeros((1, K), np.uint16)
        x[0, k] = one
        y = oracle.linear_bf16(x, W)
        expect = [float(bf16_value_exact(W[n, k])) for n in range(N)]
        assert list(y[0]) == expect


def test_one_hot_selects_dequant_column_i8():
    K, N = 32, 6
    rng = np.random.default_rng(5)
    q = rng.integers(-127, 128, size=(N, K)).astype(np.int8)
    s = synth.uniform_bf16(synth.key(12), 1e-3, 1e-2, N)   # distinct scales per channel
    assert len(set(s.tolist())) == N
    one = bf16_of_int(1)
    for k in range(K):
        x = np.zeros((1, K), np.uint16)
        x[0, k] = one
        y = oracle.linear_i8(x, q, s)
        for n in range(N):
            assert Fraction(y[0, n]) == bf16_value_exact(s[n]) * int(q[n, k])


def test_identity_and_zero_weights():
    K = 40
    x = synth.normal_bf16(synth.key(13), 1.0, 3 * K).reshape(3, K)
    eye = np.zeros((K, K), np.uint16)
    eye[np.arange(K), np.arange(K)] = bf16_of_int(1)
    y = oracle.linear_bf16(x, eye)
    xv = (x.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    assert np.array_equal(y, xv)
    assert np.all(oracle.linear_bf16(x, np.zeros((7, K), np.uint16)) == 0)
    q0 = np.zeros((5, K), np.int8)
    s = synth.uniform_bf16(synth.key(14), 1e-3, 1e-2, 5)
    assert np.all(oracle.linear_i8(x, q0, s) == 0)


# ---------------------------------------------------------------- linearity
def test_linearity_disjoint_support_and_homogeneity():
    K, N = 64, 9
    W = synth.normal_bf16(synth.key(15), 0.125, N * K).reshape(N, K)
    x = synth.normal_bf16(synth.key(16), 1.0, K).reshape(1, K)
    even = x.copy()
    even[0, 1::2] = 0
    odd = x.copy()
    odd[0, 0::2] = 0
    y, ye, yo = (oracle.linear_bf16(v, W) for v in (x, even, odd))
    assert np.allclose(y, ye + yo, rtol=1e-12, atol=1e-14)
    # homogeneity with a power of two: scaling bf16 x by 2 is exact (exponent + 1)
    x2 = x.copy()
    nz = (x2 & 0x7F80) != 0
    x2[nz] = x2[nz] + 0x80
    assert np.array_equal(oracle.linear_bf16(x2, W), 2 * y)
    # negation flips the sign bit and the output
    assert np.array_equal(oracle.linear_bf16(x ^ 0x8000, W), -y)


# ---------------------------------------------------------------- exact dequant of known codes
def test_exact_dequant_known_codes():
    # s = 2^-7 exactly in bf16 (0x3C00); q = -127 -> -127/128
    assert oracle.bf16_to_double(0x3C00) == 2.0 ** -7
    # bf16(0.005) = 0x3BA4 = 0.0050048828125 exactly
    assert oracle.bf16_to_double(0x3BA4) == 0.0050048828125
    q = np.array([[-127, -1, 0, 1, 127]], np.int8)
    for sb in (0x3C00, 0x3BA4, 0x3A83, 0x3C24, 0x3F80):
        Wd = oracle.dequant_i8(q, np.array([sb], np.uint16))
        for j, c in enumerate(q[0]):
            assert Fraction(Wd[0, j]) == bf16_value_exact(sb) * int(c)
    Wd = oracle.dequant_i8(np.array([[-127, 127]], np.int8), np.array([0x3C00], np.uint16))
    assert Wd[0, 0] == -0.9921875
    Wd = oracle.dequant_i8(np.array([[127]], np.int8), np.array([0x3BA4], np.uint16))
    assert Wd[0, 0] == 0.6356201171875


def test_bf16_decode_matches_ieee_layout():
    rng = np.random.default_rng(3)
    for h in rng.integers(0, 0x7F80, size=200).tolist() + [0, 1, 0x0080, 0x7F7F]:
        for sgn in (0, 0x8000):
            assert Fraction(oracle.bf16_to_double(h | sgn)) == bf16_value_exact(h | sgn)


# ---------------------------------------------------------------- fp64 error bound vs exact sums
@pytest.mark.parametrize("K", [16, 64, 256])
def test_error_bound_against_exact_rational_sum(K):
    N = 6
    x = synth.normal_bf16(synth.key(20, K), 1.0, 2 * K).reshape(2, K)
    W = synth.normal_bf16(synth.key(21, K), 1.0 / np.sqrt(K), N * K).reshape(N, K)
    y = oracle.linear_bf16(x, W)
    u = 2.0 ** -53
    gamma = K * u / (1 - K * u)
    for m in range(2):
        for n in range(N):
            terms = [bf16_value_exact(x[m, k]) * bf16_value_exact(W[n, k]) for k in range(K)]
            exact = sum(terms)
            absum = sum(abs(t) for t in terms)
            assert abs(Fraction(y[m, n]) - exact) <= Fraction(gamma) * absum


def test_i8_error_bound_against_exact_rational_sum():
    K, N = 128, 4
    x = synth.normal_bf16(synth.key(22), 1.0, K).reshape(1, K)
    q = synth.codes_i8(synth.key(23), N * K).reshape(N, K)
    s = synth.uniform_bf16(synth.key(24), 1e-3, 1e-2, N)
    y = oracle.linear_i8(x, q, s)
    u = 2.0 ** -53
    gamma = (K + 1) * u / (1 - (K + 1) * u)
    for n in range(N):
        terms = [bf16_value_exact(x[0, k]) * bf16_value_exact(s[n]) * int(q[n, k]) for k in range(K)]
        assert abs(Fraction(y[0, n]) - sum(terms)) <= Fraction(gamma) * sum(abs(t) for t in terms)


# ---------------------------------------------------------------- statistics of the workload recipe
def test_output_variance_is_one_for_recipe():
    W_ = wl.WORKLOADS["linear-2048"]
    p = W_.projs[0]
    x = wl.gen_x(0, W_, p).reshape(1, p.K)
    W = wl.gen_w_bf16(0, W_, p).reshape(p.N, p.K)
    y = oracle.linear_bf16(x, W)
    # Var(y_n | x) = |x|^2 / K ~ 1 for x ~ N(0,1), W ~ N(0,1/K)
    assert 0.85 < y.var() < 1.15


def test_thread_count_independence(tmp_path):
    # same result with one thread: ascending-k sums per output do not depend on scheduling
    import subprocess, sys, json
    code = (
        "import numpy as np, oracle, synth, json;"
        "x=synth.normal_bf16(synth.key(30),1.0,3*300).reshape(3,300);"
        "W=synth.normal_bf16(synth.key(31),0.1,50*300).reshape(50,300);"
        "print(json.dumps(oracle.linear_bf16(x,W).ravel().tolist()))")
    env = dict(os.environ, OMP_NUM_THREADS="1", PYTHONPATH=os.path.dirname(os.path.dirname(__file__)))
    out1 = json.loads(subprocess.check_output([sys.executable, "-c", code], env=env))
    env["OMP_NUM_THREADS"] = "4"
    out4 = json.loads(subprocess.check_output([sys.executable, "-c", code], env=env))
    assert out1 == out4
