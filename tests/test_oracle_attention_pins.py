"""Pins for the oracle's decode attention (CPU): facts fixed by the definition of softmax attention.

  * one position: the output is that position's value vector, exactly;
  * identical keys: the weights are uniform, so the output is the mean of the value vectors
    (exact for small-integer values and a power-of-two count);
  * one dominant key (score 1000 above the rest): the output is its value vector (the others'
    weights, e^-1000, vanish in double);
  * the 1/sqrt(d) scale: two keys whose scores differ by 2 sqrt(d) ln 3 before scaling get weights
    3/4 and 1/4;
  * causality among the new tokens: token m sees positions up to L - M + m only;
  * invariance under a permutation of the positions (M = 1) and under a shift of every score.
A missing scale, a causal limit off by one or a missing normalisation each fails one of them
(tests/test_oracle_mutants.py).
"""
import math
import struct

import numpy as np

import oracle


def bf(v):
    b = struct.unpack("<I", struct.pack("<f", float(v)))[0]
    assert b & 0xFFFF == 0, v
    return b >> 16


def bf_arr(a):
    return np.vectorize(bf, otypes=[np.uint16])(np.asarray(a, dtype=np.float64))


def test_single_position():
    d = 8
    rng = np.random.default_rng(0)
    k = bf_arr(rng.integers(-4, 5, size=(2, 1, d)))
    v = bf_arr(rng.integers(-4, 5, size=(2, 1, d)))
    q = rng.normal(size=(1, 2 * d)).astype(np.float32)
    out = oracle.attention(q, k, v, 1)
    vals = (v.astype(np.uint32) << 16).view(np.float32)
    assert np.array_equal(out[0], vals.reshape(-1).astype(np.float64))


def test_identical_keys_average_values():
    d, L = 16, 8
    rng = np.random.default_rng(1)
    k = np.broadcast_to(bf_arr(rng.integers(-3, 4, size=d)), (1, L, d)).copy()
    vi = rng.integers(-8, 9, size=(1, L, d))
    v = bf_arr(vi)
    q = rng.normal(size=(1, d)).astype(np.float32)
    out = oracle.attention(q, k, v, L)
    assert np.array_equal(out[0], vi[0].mean(axis=0))


def test_dominant_key_selects_its_value():
    d, L = 4, 6
    k = np.zeros((1, L, d), np.uint16)
    k[0, 3, 0] = bf(2.0)
    v = bf_arr(np.arange(L * d).reshape(1, L, d))
    q = np.zeros((1, d), np.float32)
    q[0, 0] = 1000.0                       # score 2000 / sqrt(4) = 1000 above every other key
    out = oracle.attention(q, k, v, L)
    assert np.array_equal(out[0], np.arange(3 * d, 4 * d, dtype=np.float64))


def test_scale_one_over_sqrt_d():
    d, L = 16, 2
    k = np.zeros((1, L, d), np.uint16)
    k[0, 0, 0] = bf(1.0)
    v = np.zeros((1, L, d), np.uint16)
    v[0, 0, 0] = bf(1.0)
    v[0, 1, 1] = bf(1.0)
    q = np.zeros((1, d), np.float32)
    q[0, 0] = np.float32(math.sqrt(d) * math.log(3))       # scaled score difference ln 3 (in fp32)
    t = float(q[0, 0]) / math.sqrt(d)
    out = oracle.attention(q, k, v, L)
    w0 = 1 / (1 + math.exp(-t))
    assert abs(out[0, 0] - w0) < 1e-15 and abs(out[0, 1] - (1 - w0)) < 1e-15
    assert abs(w0 - 0.75) < 1e-7


def test_causal_among_new_tokens():
    d, L, M = 4, 5, 3
    k = np.zeros((1, L, d), np.uint16)
    v = bf_arr(np.arange(L * d).reshape(1, L, d) % 7)
    q = np.zeros((M, d), np.float32)
    for j in range(L):
        k[0, j, 0] = bf(float(j))              # later positions score higher
    q[:, 0] = 1e5                              # adjacent positions' scores differ by 5e4
    out = oracle.attention(q, k, v, L)
    vals = (v.astype(np.uint32) << 16).view(np.float32)[0].astype(np.float64)
    for m in range(M):
        assert np.array_equal(out[m], vals[L - M + m]), m   # each token's newest visible position wins


def test_permutation_and_shift_invariance():
    d, L = 32, 40
    rng = np.random.default_rng(2)
    k = bf_arr(rng.integers(-8, 9, size=(2, L, d)) / 8)
    v = bf_arr(rng.integers(-8, 9, size=(2, L, d)) / 4)
    q = rng.normal(size=(1, 2 * d)).astype(np.float32)
    out = oracle.attention(q, k, v, L)
    perm = rng.permutation(L)
    out_p = oracle.attention(q, k[:, perm], v[:, perm], L)
    assert np.allclose(out, out_p, rtol=1e-13, atol=1e-13)
    # every key gains the same component along a direction q also gains: every score shifts equally
    k2 = k.copy()
    k2[:, :, -1] = bf(1.0)
    q2 = q.copy()
    q2[0, d - 1] = 0.0
    q2[0, 2 * d - 1] = 0.0
    base = oracle.attention(q2, k2, v, L)
    q2[0, d - 1] = 5.0
    q2[0, 2 * d - 1] = -3.0
    shifted = oracle.attention(q2, k2, v, L)
    assert np.allclose(base, shifted, rtol=1e-13, atol=1e-13)
