"""GPU parity of prompt-lookup decoding around the verification pass (aio_pld_draft, aio_argmax_rows,
aio_pld_accept) against oracle/pld.py, and of the routing decision (aio_route) against
oracle/route.py.  Drafting, argmax and acceptance are integer or comparison work, so the bar is
bit-exact: the same draft length, matched n, position and tokens; the same argmax index; the same
accepted count and next token.  Cases: sequences with many repeats (small vocabularies) and few
(large), lengths from 1 to the paper's 32K context, every look-ahead up to 7, windows up to 32;
logits with planted ties and NaNs, ragged vocabulary sizes and row strides; every acceptance
prefix; argument errors raised before any launch.
"""
import numpy as np
import pytest
import torch

from oracle import pld

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def aio():
    from paper_2604_09752_gb300 import aio as mod
    assert torch.cuda.is_available()
    return mod


def gpu_draft(aio, toks, N, L):
    t = torch.tensor(toks, dtype=torch.int32, device="cuda")
    out = torch.full((3 + L,), 12345, dtype=torch.int32, device="cuda")
    aio.aio_pld_draft(t.data_ptr(), len(toks), N, L, out.data_ptr(), torch.cuda.current_stream().cuda_stream)
    o = out.cpu().tolist()
    return o[3: 3 + o[0]], o[1], o[2], o


@pytest.mark.parametrize("T,vocab", [(1, 3), (2, 2), (7, 3), (100, 4), (2048, 50), (2048, 32000), (32768, 8),
                                     (32768, 32000)])
@pytest.mark.parametrize("L", [1, 2, 7])
def test_draft_matches_oracle(aio, T, vocab, L):
    rng = np.random.default_rng(T * 7 + vocab + L)
    toks = rng.integers(0, vocab, size=T).tolist()
    if T >= 64 and vocab > 100:
        toks[-6:] = toks[T // 3: T // 3 + 6]        # plant a 6-gram repeat in a sparse sequence
    d, n, i, raw = gpu_draft(aio, toks, 6, L)
    d_ref, n_ref, i_ref = pld.draft(toks, 6, L)
    assert (d, n, i) == (d_ref, n_ref, i_ref)
    assert raw[3 + len(d):] == [-1] * (L - len(d))


@pytest.mark.parametrize("N", [1, 3, 32])
def test_draft_window_sizes(aio, N):
    rng = np.random.default_rng(N)
    toks = rng.integers(0, 3, size=500).tolist()
    d, n, i, _ = gpu_draft(aio, toks, N, 2)
    assert (d, n, i) == pld.draft(toks, N, 2)


@pytest.mark.parametrize("M,V,stride", [(1, 32000, 32000), (3, 32000, 32000), (8, 37, 40), (2, 1, 1)])
def test_argmax_matches_oracle(aio, M, V, stride):
    rng = np.random.default_rng(M * 100 + V)
    x = rng.integers(-50, 50, size=(M, stride)).astype(np.float32)    # integer logits: many ties
    if V > 10:
        x[0, V // 2] = x[0, :V].max()                                  # a tie with an earlier maximum
        x[-1, 5] = np.nan                                              # NaN counts as the maximum
    xd = torch.from_numpy(x).cuda()
    out = torch.full((M,), -7, dtype=torch.int32, device="cuda")
    aio.aio_argmax_rows(xd.data_ptr(), M, V, stride, out.data_ptr(), torch.cuda.current_stream().cuda_stream)
    assert out.cpu().numpy().tolist() == pld.argmax(x[:, :V]).tolist()


def test_accept_every_prefix(aio):
    draft_buf = torch.tensor([2, 2, 10, 4, 9], dtype=torch.int32, device="cuda")   # d = 2, draft [4, 9]
    for rows, want in [([4, 9, 2], (2, 2)), ([4, 7, 2], (1, 7)), ([3, 9, 2], (0, 3))]:
        am = torch.tensor(rows, dtype=torch.int32, device="cuda")
        res = torch.zeros(2, dtype=torch.int32, device="cuda")
        aio.aio_pld_accept(am.data_ptr(), draft_buf.data_ptr(), res.data_ptr(), 0)
        assert tuple(res.cpu().tolist()) == want == pld.accept(rows, [4, 9])
    empty = torch.tensor([0, 0, -1, -1, -1], dtype=torch.int32, device="cuda")
    am = torch.tensor([5], dtype=torch.int32, device="cuda")
    res = torch.zeros(2, dtype=torch.int32, device="cuda")
    aio.aio_pld_accept(am.data_ptr(), empty.data_ptr(), res.data_ptr(), 0)
    assert tuple(res.cpu().tolist()) == (0, 5)


def test_draft_verify_accept_round_trip(aio):
    """draft -> verification logits that agree with the first drafted token only -> accept."""
    rng = np.random.default_rng(9)
    toks = rng.integers(0, 20, size=1000).tolist()
    toks[-6:] = toks[100:106]
    d, n, i, _ = gpu_draft(aio, toks, 6, 2)
    assert len(d) == 2
    V = 20
    logits = np.zeros((3, V), np.float32)
    logits[0, d[0]] = 1.0                 # agrees with draft[0]
    logits[1, (d[1] + 1) % V] = 1.0       # disagrees with draft[1]
    logits[2, 3] = 1.0
    ld = torch.from_numpy(logits).cuda()
    am = torch.zeros(3, dtype=torch.int32, device="cuda")
    aio.aio_argmax_rows(ld.data_ptr(), 3, V, V, am.data_ptr(), 0)
    t = torch.tensor(toks, dtype=torch.int32, device="cuda")
    dbuf = torch.zeros(5, dtype=torch.int32, device="cuda")
    aio.aio_pld_draft(t.data_ptr(), len(toks), 6, 2, dbuf.data_ptr(), 0)
    res = torch.zeros(2, dtype=torch.int32, device="cuda")
    aio.aio_pld_accept(am.data_ptr(), dbuf.data_ptr(), res.data_ptr(), 0)
    assert tuple(res.cpu().tolist()) == pld.accept(pld.argmax(logits).tolist(), d) == (1, (d[1] + 1) % V)


def test_argument_errors(aio):
    buf = torch.zeros(4096, dtype=torch.int32, device="cuda")
    p = buf.data_ptr()
    for args, status in [((p, 0, 6, 2, p + 64), aio.AIO_ERR_INVALID_ARG), ((p, 10, 0, 2, p + 64), aio.AIO_ERR_INVALID_ARG),
                         ((p, 10, 33, 2, p + 64), aio.AIO_ERR_INVALID_ARG), ((p, 10, 6, 8, p + 64), aio.AIO_ERR_INVALID_ARG),
                         ((p + 2, 10, 6, 2, p + 64), aio.AIO_ERR_ALIGNMENT), ((0, 10, 6, 2, p + 64), aio.AIO_ERR_INVALID_ARG)]:
        with pytest.raises(aio.AioError) as e:
            aio.aio_pld_draft(*args, 0)
        assert e.value.status == status
    for args, status in [((p, 0, 10, 10, p + 64), aio.AIO_ERR_INVALID_ARG), ((p, 1, 10, 9, p + 64), aio.AIO_ERR_INVALID_ARG),
                         ((p + 1, 1, 10, 10, p + 64), aio.AIO_ERR_ALIGNMENT)]:
        with pytest.raises(aio.AioError) as e:
            aio.aio_argmax_rows(*args, 0)
        assert e.value.status == status


def entropy_f32_bound(n, H):
    """First-order error bound of the kernel's float32 softmax entropy over n categories: each p_c
    carries ~(n + 4) ulps from exp, the n-term sum and the division, ln p_c one more, and the n-term
    sum of p_c ln p_c n more; |dH| <= (2n + 8) 2^-24 (1 + H) covers all of them."""
    return (2 * n + 8) * 2.0 ** -24 * (1.0 + H)


# Decisions whose exact entropy lies within this distance of tau are not compared: there the float32
# and the double entropy may fall on either side.  It is more than 10x entropy_f32_bound(32, tau).
ROUTE_BAND = 1e-4


def test_route_matches_oracle(aio):
    """aio_route against oracle/route.py (the entropy in double, the plain definition): the category
    and the PLD switch exactly, the model exactly outside ROUTE_BAND around tau, the float32 entropy
    within entropy_f32_bound of the double one."""
    from oracle import route
    rng = np.random.default_rng(3)
    V = 32000
    cases = 0
    for trial in range(200):
        n = int(rng.choice([2, 3, 5, 32]))
        cat_tok = rng.choice(V, size=n, replace=False).astype(np.int32)
        logits = rng.normal(scale=float(rng.choice([0.5, 2.0, 6.0])), size=V).astype(np.float32)
        code = int(rng.integers(0, n))
        L_ctx = int(rng.choice([0, 100, 2047, 2048, 2049, 32768]))
        ld = torch.from_numpy(logits).cuda()
        td = torch.from_numpy(cat_tok).cuda()
        dec = torch.zeros(4, dtype=torch.int32, device="cuda")
        aio.aio_route(ld.data_ptr(), td.data_ptr(), n, code, L_ctx, 0.45, dec.data_ptr(), 0)
        c, m, pld_on, hbits = dec.cpu().tolist()
        H = float(np.array([hbits], np.int32).view(np.float32)[0])
        c_ref, H_ref, m_ref, pld_ref = route.route(logits[cat_tok], code, L_ctx)
        assert c == c_ref and bool(pld_on) == pld_ref
        assert abs(H - H_ref) <= entropy_f32_bound(n, H_ref), (n, H, H_ref)
        if abs(H_ref - 0.45) > ROUTE_BAND:
            assert m == m_ref
            cases += 1
    assert cases > 150
