"""GPU parity of decode attention over a KV cache (aio_attention_decode) against the fp64 oracle.

Bar (per call, over out [M, n_heads * 128]): relative L2 <= 1e-3 and max |err| <= 1e-2 max |ref|,
the projections' bar.  The kernel computes in fp32 (scores from 128 products, an online softmax
in base 2, sums over up to 32K positions), whose error is orders of magnitude below it.  Cases
cover ragged caches (L not a multiple of the 16-position unit, L < 16, a single position), every
M up to 8 with the causal limit among the new tokens, q rows wider than the heads (q read from a
QKV output), flat and peaked attention, the 7B-class shapes at the paper's 2K and 32K contexts,
reproducibility, and argument errors raised before any launch.
"""
import numpy as np
import pytest
import torch

import oracle
import parity
import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def aio():
    from paper_2604_09752_gb300 import aio as mod
    assert torch.cuda.is_available()
    return mod


def make_case(n_heads, L_max, M, q_stride, seed, q_scale=1.0):
    d = 128
    k = synth.normal_bf16(synth.key(seed, 1), 1.0, n_heads * L_max * d).reshape(n_heads, L_max, d)
    v = synth.normal_bf16(synth.key(seed, 2), 1.0, n_heads * L_max * d).reshape(n_heads, L_max, d)
    qb = synth.normal_bf16(synth.key(seed, 3), 1.0, M * q_stride).reshape(M, q_stride)
    q = ((qb.astype(np.uint32) << 16).view(np.float32) * np.float32(q_scale)).astype(np.float32)
    return q, k, v


def run(aio, q, k, v, L, M, n_heads):
    d = 128
    L_max = k.shape[1]
    qd = torch.from_numpy(q).cuda()
    kd = torch.from_numpy(k.view(np.int16)).cuda()
    vd = torch.from_numpy(v.view(np.int16)).cuda()
    out = torch.full((M, n_heads * d), float("nan"), dtype=torch.float32, device="cuda")
    wsb = aio.aio_attention_workspace_bytes(M)
    ws = torch.zeros(wsb, dtype=torch.uint8, device="cuda")
    aio.aio_attention_decode(qd.data_ptr(), q.shape[1], kd.data_ptr(), vd.data_ptr(), n_heads, d, L_max, L, M,
                             out.data_ptr(), ws.data_ptr(), wsb, torch.cuda.current_stream().cuda_stream)
    assert aio.aio_attention_check(ws.data_ptr()) == 0
    return out.cpu().numpy()


def check(out, ref, what):
    out = out.astype(np.float64)
    assert np.all(np.isfinite(out)), f"{what}: non-finite output"
    rel = np.linalg.norm(out - ref) / np.linalg.norm(ref)
    assert rel <= parity.REL_L2, f"{what}: relative L2 {rel:.3e}"
    mx = np.abs(out - ref).max() / np.abs(ref).max()
    assert mx <= parity.MAX_REL, f"{what}: max error {mx:.3e} of max |ref|"
    return rel


@pytest.mark.parametrize("L", [1, 5, 16, 37, 64])
@pytest.mark.parametrize("M", [1, 2, 3, 8])
def test_small_caches(aio, L, M):
    if M > L:
        pytest.skip("M new tokens need L >= M")
    n_heads, L_max = 4, 64
    q, k, v = make_case(n_heads, L_max, M, n_heads * 128, seed=L * 10 + M)
    ref = oracle.attention(q, k, v, L)
    check(run(aio, q, k, v, L, M, n_heads), ref, f"L={L} M={M}")


@pytest.mark.parametrize("q_scale", [1.0, 8.0])
def test_wide_q_rows_and_peaked_attention(aio, q_scale):
    n_heads, L_max, L, M = 8, 300, 291, 3
    q, k, v = make_case(n_heads, L_max, M, 3 * n_heads * 128, seed=7, q_scale=q_scale)   # q inside QKV rows
    ref = oracle.attention(q, k, v, L)
    check(run(aio, q, k, v, L, M, n_heads), ref, f"q_scale={q_scale}")


@pytest.mark.parametrize("L,M", [(2048, 1), (2048, 3), (32768, 1), (32768, 3)])
def test_7b_heads_at_paper_contexts(aio, L, M):
    n_heads = 32
    q, k, v = make_case(n_heads, L, M, n_heads * 128, seed=L + M)
    ref = oracle.attention(q, k, v, L)
    check(run(aio, q, k, v, L, M, n_heads), ref, f"7B heads L={L} M={M}")


def test_reproducible(aio):
    n_heads, L_max, L, M = 32, 2048, 2000, 2
    q, k, v = make_case(n_heads, L_max, M, n_heads * 128, seed=11)
    a = run(aio, q, k, v, L, M, n_heads)
    b = run(aio, q, k, v, L, M, n_heads)
    assert np.array_equal(a.view(np.uint32), b.view(np.uint32))


def test_argument_errors(aio):
    buf = torch.zeros(1 << 22, dtype=torch.uint8, device="cuda")
    p = buf.data_ptr()
    wsb = aio.aio_attention_workspace_bytes(1)
    ws = torch.zeros(wsb, dtype=torch.uint8, device="cuda").data_ptr()
    good = dict(q=p, q_stride=512, k=p + 65536, v=p + 131072, n_heads=4, head_dim=128, L_max=16, L=16, M=1,
                out=p + 262144, ws=ws, wsb=wsb)
    cases = [(dict(head_dim=64), aio.AIO_ERR_UNSUPPORTED), (dict(M=9), aio.AIO_ERR_INVALID_ARG),
             (dict(L=17), aio.AIO_ERR_INVALID_ARG), (dict(L=0), aio.AIO_ERR_INVALID_ARG),
             (dict(q_stride=256), aio.AIO_ERR_INVALID_ARG), (dict(q=p + 4), aio.AIO_ERR_ALIGNMENT),
             (dict(q_stride=514), aio.AIO_ERR_ALIGNMENT), (dict(wsb=wsb - 16), aio.AIO_ERR_INVALID_ARG),
             (dict(k=0), aio.AIO_ERR_INVALID_ARG), (dict(n_heads=100000, q_stride=100000 * 128), aio.AIO_ERR_UNSUPPORTED)]
    for change, status in cases:
        a = dict(good, **change)
        with pytest.raises(aio.AioError) as e:
            aio.aio_attention_decode(a["q"], a["q_stride"], a["k"], a["v"], a["n_heads"], a["head_dim"], a["L_max"],
                                     a["L"], a["M"], a["out"], a["ws"], a["wsb"], 0)
        assert e.value.status == status, (change, e.value)
