"""Pins for the oracle's chained-step functions (CPU): facts fixed by arithmetic, not by the oracle.

The steps between projections of a chained decoder step (the reading of the paper's decoder,
whose block structure Sec. 4.2 does not print) are bf16 rounding, the logistic-weighted SwiGLU,
RMSNorm with a residual add, and a column slice.  They are pinned by:
  * bf16 rounding against exact rationals (nearest, ties to even, subnormals, overflow) and
    against PyTorch's float32 -> bfloat16 conversion;
  * closed forms of silu: silu(0) = 0, silu(ln 3) = (3/4) ln 3, silu(t) - silu(-t) = t;
  * RMSNorm cases whose root mean square is rational (one-hot, constant, (3, 4, 0, 0)), its
    invariance under power-of-two scaling and its oddness, and the exact fp32 residual add;
  * SwiGLU and slice cases with exact results.
A rounding toward zero, a sign error in the logistic, a mean over K - 1, or gate and up swapped
each fails one of them (tests/test_oracle_mutants.py).
"""
import math
import struct
from fractions import Fraction

import numpy as np
import pytest

import oracle


def bf16_bits_of_f32(v):
    b = struct.unpack("<I", struct.pack("<f", float(v)))[0]
    assert b & 0xFFFF == 0, v
    return b >> 16


def bf16_exact(h):
    h = int(h)
    sign = -1 if h & 0x8000 else 1
    e, m = (h >> 7) & 0xFF, h & 0x7F
    if e == 0:
        return sign * Fraction(m, 128) * Fraction(2) ** -126
    return sign * (1 + Fraction(m, 128)) * Fraction(2) ** (e - 127)


def rne_bf16_reference(v: Fraction) -> int:
    """Nearest bf16 to the rational v, ties to the even mantissa, by search over exact values."""
    if v == 0:
        return 0
    sign = 0x8000 if v < 0 else 0
    a = abs(v)
    # largest finite bf16 is (2 - 2^-7) 2^127; halfway to 2^128 rounds to infinity
    if a >= (2 - Fraction(1, 256)) * Fraction(2) ** 127:
        return sign | 0x7F80
    lo = 0
    for hb in range(0x7F80):            # finite positive patterns in increasing value order
        if bf16_exact(hb) <= a:
            lo = hb
        else:
            break
    hi = lo + 1
    dlo, dhi = a - bf16_exact(lo), bf16_exact(hi) - a
    if dlo < dhi or (dlo == dhi and lo % 2 == 0):
        return sign | lo
    return sign | hi


def _bf16_reference_fast(v: float) -> int:
    """The same nearest-even rounding by exact rational arithmetic on the binade (no search)."""
    if v == 0:
        return 0x8000 if math.copysign(1.0, v) < 0 else 0
    f = Fraction(v)
    sign = 0x8000 if f < 0 else 0
    a = abs(f)
    e = math.floor(math.log2(a)) if a >= Fraction(2) ** -126 else -126
    while Fraction(2) ** e > a:
        e -= 1
    while Fraction(2) ** (e + 1) <= a:
        e += 1
    e = max(e, -126)
    q = Fraction(2) ** (e - 7)
    n = a / q
    fl = math.floor(n)
    rem = n - fl
    if rem > Fraction(1, 2) or (rem == Fraction(1, 2) and fl % 2 == 1):
        fl += 1
    r = fl * q
    if r >= Fraction(2) ** 128:
        return sign | 0x7F80
    bits = struct.unpack("<I", struct.pack("<f", float(r)))[0]
    assert Fraction(float(r)) == r
    return sign | (bits >> 16)


def test_bf16_rounding_search_and_fast_references_agree():
    rng = np.random.default_rng(5)
    for v in list(rng.normal(size=40)) + [1 + 2 ** -8, 1 + 3 * 2 ** -8, 2.0 ** -130, 3.0e38]:
        assert rne_bf16_reference(Fraction(float(v))) == _bf16_reference_fast(float(v))


def test_bf16_rounding_exact_rationals():
    rng = np.random.default_rng(11)
    vals = []
    for scale in (1e-30, 1e-3, 1.0, 7.0, 1e5, 1e30):
        vals += list(rng.normal(size=300) * scale)
    # ties, just-off-ties, subnormals, the overflow threshold, signed zero
    vals += [1 + 2 ** -8, 1 + 3 * 2 ** -8, -(1 + 2 ** -8), 1 + 2 ** -8 + 2 ** -40, 1 + 2 ** -8 - 2 ** -40,
             2.0 ** -133, 1.5 * 2.0 ** -133, 2.5 * 2.0 ** -133, 2.0 ** -134, 2.0 ** -135, 2.0 ** -126 * 0.75,
             (2 - 2 ** -8) * 2.0 ** 127, (2 - 2 ** -8) * 2.0 ** 127 * (1 - 2 ** -30), 1e39, -1e39, 0.0, -0.0]
    for v in vals:
        assert oracle.double_to_bf16(v) == _bf16_reference_fast(float(v)), v


def test_bf16_rounding_matches_library_for_float32_values():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(3)
    f = np.concatenate([rng.normal(size=4000).astype(np.float32) * s for s in (1e-20, 1.0, 1e20)])
    lib = torch.from_numpy(f).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    ours = np.array([oracle.double_to_bf16(float(v)) for v in f], np.uint16)
    assert np.array_equal(ours, lib)


def test_bf16_known_ties():
    assert oracle.double_to_bf16(1 + 2 ** -8) == 0x3F80          # halfway, even stays
    assert oracle.double_to_bf16(1 + 3 * 2 ** -8) == 0x3F82      # halfway, odd rounds up
    assert oracle.double_to_bf16(-(1 + 3 * 2 ** -8)) == 0xBF82
    assert oracle.double_to_bf16(1 + 2 ** -8 + 2 ** -30) == 0x3F81
    assert oracle.double_to_bf16(1e39) == 0x7F80
    assert oracle.double_to_bf16(-0.0) == 0x8000


def test_silu_closed_forms():
    assert oracle.silu(0.0) == 0.0
    assert abs(oracle.silu(math.log(3)) - 0.75 * math.log(3)) < 1e-15
    for t in (0.1, 0.5, 1.0, 2.5, 7.0, 30.0):
        assert abs((oracle.silu(t) - oracle.silu(-t)) - t) < 1e-14 * max(1.0, t)
    assert oracle.silu(-40.0) < 0 and abs(oracle.silu(-40.0)) < 1e-15
    assert abs(oracle.silu(40.0) - 40.0) < 1e-13


def _gamma(K, seed=1):
    rng = np.random.default_rng(seed)
    return np.array([bf16_bits_of_f32(struct.unpack("<f", struct.pack("<I", int(b) << 16))[0])
                     for b in (0x3F00 + rng.integers(0, 0x100, size=K))], np.uint16)   # values in [0.5, 2)


def test_rmsnorm_one_hot_and_constant():
    K = 64                                  # sqrt(K) = 8: the root mean square is rational
    g = _gamma(K)
    for k in (0, 17, 63):
        for c in (3.0, -0.75, 1e-3):
            h = np.zeros((1, K), np.float32)
            h[0, k] = c
            _, x = oracle.rmsnorm(h, None, g, 0.0)
            # x_k = c / (|c| / 8) * g_k = 8 sign(c) g_k exactly; every other entry is 0
            want = (int(g[k]) + (3 << 7)) | (0x8000 if c < 0 else 0)
            assert int(x[0, k]) == want
            assert not np.any(np.delete(x[0], k) & 0x7FFF)
    h = np.full((2, K), -2.5, np.float32)
    _, x = oracle.rmsnorm(h, None, g, 0.0)
    assert np.array_equal(x[0], g | 0x8000) and np.array_equal(x[1], g | 0x8000)


def test_rmsnorm_rational_case():
    g = np.array([bf16_bits_of_f32(v) for v in (1.0, 1.0, 0.5, 2.0)], np.uint16)
    h = np.array([[3.0, 4.0, 0.0, 0.0]], np.float32)       # mean of squares 25/4, rms 5/2
    _, x = oracle.rmsnorm(h, None, g, 0.0)
    assert [int(v) for v in x[0]] == [rne_bf16_reference(Fraction(6, 5)), rne_bf16_reference(Fraction(8, 5)), 0, 0]
    # with eps: rms = sqrt(25/4 + 39/4) = 4
    _, x = oracle.rmsnorm(h, None, g, 39 / 4)
    assert [int(v) for v in x[0]] == [rne_bf16_reference(Fraction(3, 4)), 0x3F80, 0, 0]


def test_rmsnorm_invariances_and_residual():
    rng = np.random.default_rng(7)
    K = 96
    g = _gamma(K, 2)
    h = rng.normal(size=(3, K)).astype(np.float32)
    _, x = oracle.rmsnorm(h, None, g, 0.0)
    for j in (-3, 5):
        _, xs = oracle.rmsnorm((h * np.float32(2.0 ** j)).astype(np.float32), None, g, 0.0)
        assert np.array_equal(xs, x)
    _, xn = oracle.rmsnorm(-h, None, g, 0.0)
    assert np.array_equal(xn, x ^ 0x8000)
    r = rng.normal(size=(3, K)).astype(np.float32)
    h_out, x1 = oracle.rmsnorm(h, r, g, 1e-5)
    assert np.array_equal(h_out.view(np.uint32), (h + r).view(np.uint32))   # one float32 add, nearest-even
    _, x2 = oracle.rmsnorm((h + r).astype(np.float32), None, g, 1e-5)
    assert np.array_equal(x1, x2)
    _, xz = oracle.rmsnorm(np.zeros((1, K), np.float32), None, g, 1e-5)
    assert not np.any(xz & 0x7FFF)


def test_swiglu_exact_cases():
    I = 5
    ln3 = math.log(3)
    y = np.zeros((2, 2 * I + 3), np.float32)               # stride > 2I: padding columns ignored
    y[0, :I] = [0.0, np.float32(ln3), 2.0, -1.0, 5.0]
    y[0, I:2 * I] = [7.0, 0.0, 0.0, 0.0, 0.0]
    y[0, 2 * I:] = 99.0
    y[1, :I] = np.float32(ln3)
    y[1, I:2 * I] = [np.float32(4 / (3 * float(np.float32(ln3)))), 1.0, -2.0, 0.5, 4.0]
    x = oracle.swiglu(y, I)
    assert not np.any(x[0] & 0x7FFF)                        # silu(0) = 0, and u = 0
    t = float(np.float32(ln3))
    s = t / (1 + math.exp(-t))
    for k, u in enumerate(y[1, I:2 * I]):
        assert int(x[1, k]) == _bf16_reference_fast(s * float(u))
    assert int(x[1, 0]) == 0x3F80                          # silu(ln 3) * 4 / (3 ln 3) = 1


def test_slice_exact():
    y = np.arange(3 * 40, dtype=np.float32).reshape(3, 40)
    x = oracle.slice_x(y, 24, 16)
    want = np.array([[bf16_bits_of_f32(v) for v in row[24:40]] for row in y], np.uint16)
    assert np.array_equal(x, want)


def _tiny_chain(zero_o_down: bool):
    from synth import workloads as swl
    H, I, V, L = 32, 48, 40, 2
    projs = []
    for l in range(L):
        projs += [swl.Proj(l, 0, H, 3 * H), swl.Proj(l, 1, H, H), swl.Proj(l, 2, H, 2 * I), swl.Proj(l, 3, I, H)]
    projs.append(swl.Proj(L, 4, H, V))
    wl = swl.Workload("tiny-chain", 9, "bf16", 1, projs)
    links = swl.chain_links(wl)
    rng = np.random.default_rng(4)
    to_bf16 = lambda a: np.array([oracle.double_to_bf16(float(v)) for v in a.ravel()], np.uint16).reshape(a.shape)
    weights = []
    for p in projs:
        W = rng.normal(size=(p.N, p.K)) / math.sqrt(p.K)
        if zero_o_down and p.index in (1, 3):
            W[:] = 0.0
        weights.append(to_bf16(W))
    gammas = [to_bf16(rng.uniform(0.5, 1.5, size=H)) for _ in range(2 * L + 1)]
    h0 = rng.normal(size=(2, H)).astype(np.float32)
    return wl, links, weights, gammas, h0


def test_chain_wiring_with_zero_o_and_down():
    # With O and down weights zero, every residual add adds zero: each RMSNorm sees h0, so the QKV
    # and gate+up inputs of every layer, and the lm_head input, are RMSNorm(h0) with their own weight.
    wl, links, weights, gammas, h0 = _tiny_chain(True)
    xs, ys, h = oracle.chain_step(links, weights, h0, gammas, 1e-5)
    for i, (p, link) in enumerate(zip(wl.projs, links)):
        if p.index in (0, 2, 4):
            _, want = oracle.rmsnorm(h0, None, gammas[link.gamma], 1e-5)
            assert np.array_equal(xs[i], want), p.name
        if p.index in (1, 3):
            assert not np.any(ys[i])
    assert np.array_equal(h[0], h0) and np.array_equal(h[1], h0)


def test_chain_wiring_general():
    wl, links, weights, gammas, h0 = _tiny_chain(False)
    xs, ys, h = oracle.chain_step(links, weights, h0, gammas, 1e-5)
    H = h0.shape[1]
    for i, (p, link) in enumerate(zip(wl.projs, links)):
        if p.index == 1:     # attention over one position: the V third of QKV
            assert np.array_equal(xs[i], oracle.slice_x(ys[i - 1], 2 * H, H))
        if p.index == 3:     # SwiGLU of gate+up
            assert np.array_equal(xs[i], oracle.swiglu(ys[i - 1], p.K))
    # the final residual stream is h0 plus every O and down output, added in order in fp32
    acc = h0.copy()
    for i, p in enumerate(wl.projs):
        if p.index in (1, 3):
            acc = (acc + ys[i]).astype(np.float32)
    assert np.array_equal(h[0], acc)
