"""The policy settings used by the oracles, the GPU tests and bench.py are the paper's printed ones
(tests/golden/paper_policy.txt, with its citations): the routing threshold and short-context bound
(Sec. 3.2, Sec. 3.3), the PLD window and look-ahead (Sec. 4.2), and the 2K / 32K contexts
(Sec. 5.1) that the attention measurements use (CPU)."""
import inspect
import os

from oracle import pld, route

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "paper_policy.txt")
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def golden():
    vals = {}
    for line in open(GOLDEN):
        line = line.strip()
        if line and not line.startswith("#"):
            k, v = line.split()
            vals[k] = float(v)
    return vals


def test_routing_constants():
    g = golden()
    assert route.TAU == g["route_entropy_tau"]
    assert route.SHORT_CONTEXT == g["route_short_context_tokens"]


def test_pld_defaults():
    g = golden()
    sig = inspect.signature(pld.draft)
    assert sig.parameters["N"].default == g["pld_ngram_window"]
    assert sig.parameters["L"].default == g["pld_lookahead"]


def test_bench_uses_the_papers_settings():
    g = golden()
    src = open(os.path.join(ROOT, "bench.py")).read()
    assert f"aio_pld_draft(t.data_ptr(), n, {int(g['pld_ngram_window'])}, {int(g['pld_lookahead'])}," in src
    assert f"for L, layers in (({int(g['context_standard_tokens'])}, 32), ({int(g['context_long_tokens'])}, 4))" in src
    # the kernel's 1B-route bound is the paper's 2K
    cu = open(os.path.join(ROOT, "paper_2604_09752_gb300", "csrc", "aio_pld.cu")).read()
    assert f"L_ctx <= {int(g['route_short_context_tokens'])}" in cu
