"""Byte accounting of the decode-step workloads (CPU).

The algorithmic bytes per step (every weight byte streamed once, plus int8
scales) are checked against a closed form over the projection shapes, and
the 7B-class total against the per-token traffic the paper prints in Sec. 3.1
(tests/golden/paper_traffic.txt).
"""
import os

from synth import workloads as wl

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "paper_traffic.txt")


def _golden():
    vals = {}
    for line in open(GOLDEN):
        line = line.strip()
        if line and not line.startswith("#"):
            k, v = line.split()
            vals[k] = float(v)
    return vals


def test_closed_form_bytes():
    # per layer: H*(3H') + H*H + H*2I + I*H elements; plus the lm_head H*V
    def total(L, H, I, QKV, V, esize):
        return (L * (H * QKV + H * H + H * 2 * I + I * H) + H * V) * esize
    assert wl.WORKLOADS["7b-bf16"].weight_bytes() == total(32, 4096, 11008, 12288, 32000, 2) == 13_214_154_752
    assert wl.WORKLOADS["1b-bf16"].weight_bytes() == total(22, 2048, 5632, 6144, 32000, 2) == 2_391_801_856
    n_scales = 32 * (12288 + 4096 + 22016 + 4096) + 32000
    assert wl.WORKLOADS["7b-int8"].weight_bytes() == total(32, 4096, 11008, 12288, 32000, 1) + 2 * n_scales \
        == 6_609_861_120
    assert wl.WORKLOADS["linear-2048"].weight_bytes() == 8_388_608
    assert len(wl.WORKLOADS["7b-bf16"].projs) == 129 and len(wl.WORKLOADS["1b-bf16"].projs) == 89


def test_7b_bytes_match_paper_traffic():
    g = _golden()
    b = wl.WORKLOADS["7b-bf16"].weight_bytes()
    assert abs(b / (g["7b_fp16_weight_gb"] * 1e9) - 1) < 0.10
    # 7.1 TB over 512 tokens is ~13.9 GB per token: weights dominate the per-token traffic
    per_token = g["7b_hbm_tb_per_512_tokens"] * 1e12 / 512
    assert 0.9 < b / per_token <= 1.0


def test_pld_widths_keep_weight_bytes():
    base = wl.WORKLOADS["7b-bf16"].weight_bytes()
    for M in wl.PLD_WIDTHS:
        assert wl.pld_workload(M, "bf16").weight_bytes() == base
        assert wl.pld_workload(M, "int8").weight_bytes() == wl.WORKLOADS["7b-int8"].weight_bytes()
