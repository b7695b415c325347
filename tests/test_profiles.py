"""The committed ncu traffic summary (profiles/gemv_traffic.txt) belongs to the current stream
kernel: bench.py reports it as the roofline's `traffic` only while the kernel source hash matches,
and the scaled DRAM bytes of a whole 7B step stay within 2% of the algorithmic weight bytes (no
weight is read twice; the rest is y and the split-group partial sums).  CPU only."""
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import bench  # noqa: E402
from synth import workloads as swl  # noqa: E402


def test_traffic_summary_matches_current_kernel_and_algorithmic_bytes():
    for name in ("7b-bf16", "7b-int8"):
        traffic, note = bench.committed_traffic(name, 1)
        assert traffic is not None, f"{name}: {note}"
        alg = swl.WORKLOADS[name].weight_bytes()
        assert 1.0 <= traffic / alg <= 1.02, (name, traffic, alg)
