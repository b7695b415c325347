"""The seeded input generator: definition, random access, distributions (CPU)."""
import math
import struct

import numpy as np

import synth
from synth import workloads as wl

MASK = 2**64 - 1


def _splitmix64(state):
    # the published splitmix64 step (Steele, Lea & Flood 2014)
    z = (state + 0x9E3779B97F4A7C15) & MASK
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & MASK
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & MASK
    return z ^ (z >> 31)


def test_splitmix64_matches_definition():
    for s in [0, 1, 2, 12345, 2**63, MASK]:
        assert synth.splitmix64(s) == _splitmix64(s)
    # a splitmix64 stream: bits(key, i) is the (i+1)-th output of a generator whose state starts at key
    k = 0xDEADBEEF
    state = k
    for i in range(5):
        out = _splitmix64(state)
        state = (state + 0x9E3779B97F4A7C15) & MASK
        assert synth.bits(k, i) == out


def test_splitmix64_known_vector():
    # first outputs of splitmix64 seeded with 0 (widely published reference values)
    assert synth.splitmix64(0) == 0xE220A8397B1DCDAF
    assert synth.bits(0, 1) == 0x6E789E6AA1B965F4


def _bf16_bits(f):
    return struct.unpack("<I", struct.pack("<f", f))[0]


def test_bf16_round_to_nearest_even():
    assert synth.f32_to_bf16(1.0) == 0x3F80
    assert synth.f32_to_bf16(-2.0) == 0xC000
    # exact tie below: 0x3F808000 rounds to even 0x3F80; 0x3F818000 rounds up to 0x3F82
    assert synth.f32_to_bf16(struct.unpack("<f", struct.pack("<I", 0x3F808000))[0]) == 0x3F80
    assert synth.f32_to_bf16(struct.unpack("<f", struct.pack("<I", 0x3F818000))[0]) == 0x3F82
    assert synth.f32_to_bf16(struct.unpack("<f", struct.pack("<I", 0x3F808001))[0]) == 0x3F81
    assert synth.f32_to_bf16(0.005) == 0x3BA4
    assert synth.f32_to_bf16(float("inf")) == 0x7F80


def test_random_access_and_odd_offsets():
    k = synth.key(7, 1, 2, 3)
    full = synth.normal_bf16(k, 0.5, 1001)
    for off, n in [(0, 1), (1, 10), (3, 7), (500, 501), (999, 2), (1000, 1)]:
        part = synth.normal_bf16(k, 0.5, n, off)
        assert np.array_equal(part, full[off:off + n]), (off, n)
    c = synth.codes_i8(k, 513)
    assert np.array_equal(synth.codes_i8(k, 100, 77), c[77:177])
    u = synth.uniform_bf16(k, 1e-3, 1e-2, 300)
    assert np.array_equal(synth.uniform_bf16(k, 1e-3, 1e-2, 5, 101), u[101:106])


def test_normal_moments():
    k = synth.key(0, 9, 9, 9)
    h = synth.normal_bf16(k, 1.0, 1 << 20)
    v = (h.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    assert abs(v.mean()) < 5e-3
    assert abs(v.var() - 1.0) < 1e-2
    # tails present (Box-Muller is exact in distribution)
    assert (np.abs(v) > 4).sum() > 20


def test_codes_uniform_range():
    k = synth.key(0, 1, 1, 2)
    c = synth.codes_i8(k, 255 * 400)
    assert c.min() == -127 and c.max() == 127
    counts = np.bincount(c.astype(np.int64) + 127, minlength=255)
    assert counts.min() > 300 and counts.max() < 520


def test_scales_range():
    k = synth.key(0, 1, 1, 3)
    s = synth.uniform_bf16(k, 1e-3, 1e-2, 10000)
    v = (s.astype(np.uint32) << 16).view(np.float32)
    assert v.min() >= 0.99e-3 and v.max() <= 1.01e-2


def test_workload_keys_distinct():
    W = wl.WORKLOADS["7b-bf16"]
    keys = {wl.tensor_key(0, W.family, p, kind) for p in W.projs for kind in range(4)}
    assert len(keys) == 4 * len(W.projs)


def test_w_sigma():
    W = wl.WORKLOADS["linear-2048"]
    p = W.projs[0]
    h = wl.gen_w_bf16(0, W, p, 0, 64)
    v = (h.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    assert abs(v.std() * math.sqrt(p.K) - 1.0) < 0.02


def test_gen_rows_matches_full():
    W = wl.WORKLOADS["linear-2048"]
    p = W.projs[0]
    full = wl.gen_w_bf16(0, W, p, 0, 40).reshape(40, p.K)
    rows = np.array([3, 0, 39, 17])
    sub, _ = wl.gen_rows(0, W, p, rows)
    assert np.array_equal(sub, full[rows])
