"""The GPU tests' tolerance helper (tests/parity.py) on the CPU: the magnitude sum_k |x_k w_k| that
sets the fp32 summation bound, including int8 code -128 (whose magnitude 128 does not fit int8)."""
import numpy as np

import parity
import synth


def bf16_values(bits):
    return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def test_magnitude_of_int8_codes_including_minus_128():
    K, N, M = 300, 7, 3
    x = synth.normal_bf16(synth.key(5, 1), 1.0, M * K).reshape(M, K)
    q = synth.codes_i8(synth.key(5, 2), N * K).reshape(N, K)
    q[0] = -128
    q[3, ::3] = -128
    s = synth.uniform_bf16(synth.key(5, 3), 1e-3, 1e-2, N)
    lo, hi = parity.abs_codes(q)
    assert lo.min() >= 0 and np.array_equal(lo.astype(np.int16) + hi, np.abs(q.astype(np.int16)))
    y, mag = parity.reference(x, q, s)
    w = np.abs(q.astype(np.float64)) * bf16_values(s)[:, None]
    want = np.abs(bf16_values(x)) @ w.T
    assert np.all(mag >= 0)
    assert np.allclose(mag, want, rtol=1e-12, atol=0)
    assert mag[:, 0].min() > 0 and np.allclose(mag[:, 0], np.abs(bf16_values(x)).sum(1) * 128 * bf16_values(s)[0])


def test_magnitude_of_bf16_weights():
    K, N, M = 64, 5, 2
    x = synth.normal_bf16(synth.key(6, 1), 1.0, M * K).reshape(M, K)
    W = synth.normal_bf16(synth.key(6, 2), 0.1, N * K).reshape(N, K)
    _, mag = parity.reference(x, W)
    assert np.allclose(mag, np.abs(bf16_values(x)) @ np.abs(bf16_values(W)).T, rtol=1e-12, atol=0)
