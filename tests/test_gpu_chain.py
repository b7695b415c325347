"""GPU parity of the chained decoder step: every projection's x is computed on the device from the
outputs of the projections before it (RMSNorm with the residual add, the V third of QKV for
attention over one position, SwiGLU), in the same persistent launch.

Attention over a KV cache (O's x in the chained step, when the workload has caches) is checked at
the attention bar instead (relative L2 <= 1e-3, max <= 1e-2 max |x|, at most 1% of elements off by
any ulp), and every layer's cache after the step bit for bit.

Two checks, both against the fp64 oracle:
  * step by step ("teacher forced"): the oracle recomputes each projection's x from the GPU's own
    earlier outputs and the residual stream they imply, and each y from the GPU's own x.  A
    computed x may differ from the oracle's by one bf16 ulp where the fp32 and fp64 values round
    differently (fp32 reductions and silu differ from fp64 in the last bits): at most one ulp and
    on at most 1% of the elements, except for values so small that the difference is below
    2^-24 max |x| (silu of a gate below about -87, where e^t is an fp32 subnormal); the V slice is
    exact.  Every y meets the linear-layer bar, and
    the final residual stream is bit-exact (fp32 adds in the same order).
  * end to end (small chains): the oracle's own chain, from h0, against every GPU output.  Each
    projection input is re-rounded to bf16, so an input that differs by a relative d before
    rounding differs after it by one ulp (2^-8 relative) on a fraction ~d / 2^-8 of its elements:
    rounding turns small differences into ulp flips, and they compound from projection to
    projection (the O input of layer 1 is the fifth re-rounding).  The step-by-step check above is
    the parity of each computation; this one bounds the drift of a two-layer chain at a relative L2
    of 1e-2 and a max error of 5e-2 max |y|, ten and five times the single-projection bar.
"""
import numpy as np
import pytest
import torch

import oracle
import parity
from synth import workloads as swl

pytestmark = pytest.mark.gpu

CHAIN_REL_L2 = 1e-2     # end-to-end drift of a two-layer chain (see the module docstring)
CHAIN_MAX_REL = 5e-2


@pytest.fixture(scope="module")
def aio():
    from paper_2604_09752_gb300 import aio as mod
    assert torch.cuda.is_available()
    return mod


def ordered(bits):
    """bf16 bit patterns as integers that step by one per ulp across zero."""
    b = bits.astype(np.int32)
    mag = b & 0x7FFF
    return np.where(b & 0x8000, -mag, mag)


def bf16_values(bits):
    return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def check_x(x_gpu, x_ref, op, what):
    if op == swl.XOP_SLICE:
        assert np.array_equal(x_gpu, x_ref), f"{what}: sliced x differs"
        return
    if op == swl.XOP_ATTENTION:
        # out = sum_j p_j v_j can cancel to values far below max |x|, where the fp32 softmax and sums
        # (errors ~2^-24 max |v| absolute) move the bf16 rounding by several ulps: the attention bar
        # of test_gpu_attention.py (the projections' bar) applies, with ulp flips still rare
        g, r = bf16_values(x_gpu), bf16_values(x_ref)
        rel = np.linalg.norm(g - r) / np.linalg.norm(r)
        assert rel <= parity.REL_L2, f"{what}: attention x relative L2 {rel:.3e}"
        mx = np.abs(g - r).max()
        assert mx <= parity.MAX_REL * np.abs(r).max(), f"{what}: attention x max error {mx:.3e}"
        flips = ordered(x_gpu) != ordered(x_ref)
        assert flips.mean() <= 0.01, f"{what}: {flips.mean():.3%} of attention x elements differ"
        return
    d = np.abs(ordered(x_gpu) - ordered(x_ref))
    tiny = np.abs(bf16_values(x_gpu) - bf16_values(x_ref)) <= 2.0 ** -24 * np.abs(bf16_values(x_ref)).max()
    bad = (d > 1) & ~tiny
    assert not bad.any(), f"{what}: x differs by {d[bad].max()} ulp at {np.argwhere(bad)[0].tolist()}"
    flips = (d > 0) & ~tiny
    assert flips.mean() <= 0.01, f"{what}: {flips.mean():.3%} of x elements differ by one ulp"


def weights_of(dw, p, rows=None):
    if rows is None:
        if dw.i8:
            return swl.gen_codes(dw.seed, dw.wl, p).reshape(p.N, p.K), swl.gen_scales(dw.seed, dw.wl, p)
        return swl.gen_w_bf16(dw.seed, dw.wl, p).reshape(p.N, p.K), None
    return swl.gen_rows(dw.seed, dw.wl, p, rows)


def kv_caches(dw, L_past):
    """The oracle's view of every layer's cache before the step: layer -> [kv bits, L_past, n_heads]."""
    if dw.kv_len is None:
        return None
    return {l: [swl.gen_kv_cache(dw.seed, dw.wl, l, dw.kv_len).reshape(2, dw.n_heads, dw.kv_len, swl.HEAD_DIM),
                L_past, dw.n_heads] for l in dw.attn_layers}


def teacher_forced(dw, M, what, rows_of=None, L_past=None):
    """Check every projection of one chained step from the GPU's own earlier outputs (and, with KV
    caches, every layer's cache after the step, bit for bit)."""
    h0 = swl.gen_h0(dw.seed, dw.wl, M)
    gammas = [dw.gamma(j).cpu().numpy().view(np.uint16) for j in range(dw.n_norms)]
    caches = kv_caches(dw, L_past)
    ys, h = [], [None, None]
    for i, (b, link) in enumerate(zip(dw.bufs, dw.links)):
        p = b.proj
        x_ref, h_out = oracle.Oracle(oracle._l()).prep(link, ys, h, h0, gammas, swl.RMS_EPS, caches)
        if h_out is not None:
            h[link.h_out] = h_out
        x_gpu = dw.x(i, M).cpu().numpy().view(np.uint16)
        check_x(x_gpu, x_ref, link.op, f"{what} {p.name} x")
        rows = rows_of(p) if rows_of else None
        W, s = weights_of(dw, p, rows)
        y_ref, mag = parity.reference(x_gpu, W, s)
        y_all = dw.y(i, M)
        assert bool(torch.isfinite(y_all).all()), f"{what} {p.name}: an output was not written"
        y_gpu = y_all.cpu().numpy()
        parity.check(y_gpu if rows is None else y_gpu[:, rows], y_ref, mag, p.K, f"{what} {p.name} y")
        ys.append(y_gpu)
    # the residual buffers hold the last values written, bit for bit
    for j in (0, 1):
        last = max((i for i, l in enumerate(dw.links) if l.h_out == j), default=None)
        if last is not None:
            assert np.array_equal(dw.h(j, M).cpu().numpy().view(np.uint32), h[j].view(np.uint32)), f"{what} h{j}"
    for layer, (kv_ref, _, _) in (caches or {}).items():
        kv_gpu = dw.kv(layer).cpu().numpy().view(np.uint16)
        assert np.array_equal(kv_gpu, kv_ref), f"{what}: layer {layer}'s KV cache after the step"
    return ys


def narrow_chain(wtype):
    """Two layers of a decoder with hidden 2048 and intermediate 2048 (QKV 6144, vocabulary 4096):
    every computed x fits the staging area at M = 4, which the 1B and 7B down projections (K = 5632,
    11008) do not."""
    return swl.Workload(f"narrow-{wtype}", 2, wtype, 1, swl.decoder(2, 2048, 2048, 6144, 4096),
                        "two-layer narrow decoder for chained M = 4")


@pytest.mark.parametrize("name,M", [("1b-bf16", 1), ("1b-bf16", 2), ("1b-bf16", 3), ("1b-bf16", 4), ("7b-int8", 1),
                                    ("7b-bf16", 1), ("7b-bf16", 3), ("7b-int8", 2), ("narrow-bf16", 4),
                                    ("narrow-int8", 4), ("narrow-bf16", 3)])
def test_small_chain(aio, name, M):
    from paper_2604_09752_gb300.workload import DeviceWorkload
    if name.startswith("narrow-"):
        wl = narrow_chain(name.split("-")[1])
    else:
        wl = swl.truncated(swl.WORKLOADS[name], 2)
    dw = DeviceWorkload(wl, seed=3, max_M=M, chained=True)
    dw.fill_chain(M)
    dw.x_arena.fill_(0xFF)
    dw.y_arena.fill_(0xFF)
    for flags in (aio.AIO_STEP_GRAPH | aio.AIO_STEP_PERSISTENT, aio.AIO_STEP_GRAPH | aio.AIO_STEP_PDL):
        dw.step(M, flags)
        dw.step(M, flags)                            # a second step starts from the same inputs
        assert aio.aio_decode_step_check(dw.step_handle(M, flags)) == 0
        ys = teacher_forced(dw, M, f"{name} M={M} flags={flags}")
    # end to end: the oracle's own chain from h0
    weights = [weights_of(dw, b.proj) for b in dw.bufs]
    weights = [w if s is None else (w, s) for w, s in weights]
    gammas = [dw.gamma(j).cpu().numpy().view(np.uint16) for j in range(dw.n_norms)]
    _, ys_ref, _ = oracle.chain_step(dw.links, weights, swl.gen_h0(dw.seed, wl, M), gammas, swl.RMS_EPS)
    drift = []
    for i, b in enumerate(dw.bufs):
        y, r = ys[i].astype(np.float64), ys_ref[i].astype(np.float64)
        rel = np.linalg.norm(y - r) / np.linalg.norm(r)
        mx = np.abs(y - r).max() / np.abs(r).max()
        drift.append(f"{b.proj.name} {rel:.2e}/{mx:.2e}")
        assert rel <= CHAIN_REL_L2, f"{name} {b.proj.name}: end-to-end relative L2 {rel:.2e}"
        assert mx <= CHAIN_MAX_REL, f"{name} {b.proj.name}: end-to-end max error {mx:.2e} of max |y|"
    print(f"{name} M={M} end-to-end drift (rel L2 / max): " + ", ".join(drift))
    dw.close()


@pytest.mark.parametrize("name,M,L_max,L_past", [
    ("7b-bf16", 1, 2048, 2047),     # the paper's 2K context, 7B-class heads (32 x 128)
    ("7b-bf16", 3, 2048, 2045),     # PLD verification of 2 drafted tokens (L = 2)
    ("7b-int8", 2, 2048, 1000),     # ragged context, int8 weights
    ("1b-bf16", 3, 64, 15),         # the new tokens straddle a 16-position unit; 16 heads
    ("1b-bf16", 1, 16, 0),          # an empty cache: attention over the new token alone
    ("narrow-int8", 4, 512, 300),   # M = 4
])
def test_chain_with_attention_over_kv_cache(aio, name, M, L_max, L_past):
    """O's x is decode attention of the new tokens over each layer's KV cache, inside the persistent
    launch (and in chain mode), checked step by step against the oracle's attention link from the
    GPU's own QKV output; the caches afterwards hold the new tokens' k and v, bit for bit."""
    from paper_2604_09752_gb300.workload import DeviceWorkload
    wl = narrow_chain(name.split("-")[1]) if name.startswith("narrow-") else swl.truncated(swl.WORKLOADS[name], 2)
    dw = DeviceWorkload(wl, seed=5, max_M=M, chained=True, kv_len=L_max)
    dw.fill_chain(M)
    dw.fill_kv(L_past)
    for flags in (aio.AIO_STEP_GRAPH | aio.AIO_STEP_PERSISTENT, aio.AIO_STEP_GRAPH | aio.AIO_STEP_PDL):
        dw.x_arena.fill_(0xFF)
        dw.y_arena.fill_(0xFF)
        dw.step(M, flags)
        dw.step(M, flags)   # a second step rewrites the same cache rows with the same values
        assert aio.aio_decode_step_check(dw.step_handle(M, flags)) == 0
        teacher_forced(dw, M, f"{name} M={M} L={L_past + M} flags={flags}", L_past=L_past)
    if L_past == 0 and M == 1:
        # attention over one position returns its value vector: x of O is the V third of QKV
        for i, l in enumerate(dw.links):
            if l.op == swl.XOP_ATTENTION:
                y = dw.y(l.src, M).cpu().numpy()
                H = dw.bufs[i].proj.K
                assert np.array_equal(dw.x(i, M).cpu().numpy().view(np.uint16), oracle.slice_x(y, 2 * H, H))
    dw.close()


def test_chain_attention_reports_a_short_cache(aio):
    """L_past + M beyond the cache: the attention phases do nothing, the step completes and reports
    device error 4; after reset, a valid L_past runs correctly again."""
    from paper_2604_09752_gb300.workload import DeviceWorkload
    wl = swl.truncated(swl.WORKLOADS["1b-bf16"], 1)
    dw = DeviceWorkload(wl, seed=6, max_M=2, chained=True, kv_len=32)
    dw.fill_chain(2)
    dw.fill_kv(31)
    dw.step(2)
    with pytest.raises(aio.AioError) as e:
        aio.aio_decode_step_check(dw.step_handle(2))
    assert e.value.status == aio.AIO_ERR_DEVICE_TIMEOUT and "code 4" in str(e.value)
    aio.aio_decode_step_reset(dw.step_handle(2))
    dw.fill_kv(20)
    dw.step(2)
    assert aio.aio_decode_step_check(dw.step_handle(2)) == 0
    teacher_forced(dw, 2, "after a short cache", L_past=20)
    dw.close()


def test_full_7b_chain_with_2k_attention_sampled(aio):
    """The whole 7B-class chained step with attention over a 2K context in every layer (32 layers
    and lm_head, M = 1, one persistent launch)."""
    from paper_2604_09752_gb300.workload import DeviceWorkload
    rng = np.random.default_rng(2)
    dw = DeviceWorkload(swl.WORKLOADS["7b-bf16"], seed=0, max_M=1, chained=True, kv_len=2048)
    dw.fill_chain(1)
    dw.fill_kv(2047)
    for _ in range(3):
        dw.step(1)
    assert aio.aio_decode_step_check(dw.step_handle(1)) == 0
    assert aio.aio_decode_step_kernels(dw.step_handle(1)) == 1

    def rows_of(p):
        return np.array(sorted({0, p.N - 1, 15, 16} | set(rng.choice(p.N, 24, replace=False).tolist())))
    teacher_forced(dw, 1, "7b chain 2K attention", rows_of, L_past=2047)
    dw.close()


def test_chain_step_is_deterministic(aio):
    from paper_2604_09752_gb300.workload import DeviceWorkload
    dw = DeviceWorkload(swl.truncated(swl.WORKLOADS["1b-bf16"], 1), seed=4, max_M=2, chained=True)
    dw.fill_chain(2)
    dw.step(2)
    torch.cuda.synchronize()
    y0, x0 = dw.y_arena.clone(), dw.x_arena.clone()
    dw.y_arena.zero_()
    dw.x_arena.zero_()
    dw.step(2)
    torch.cuda.synchronize()
    assert torch.equal(y0, dw.y_arena) and torch.equal(x0, dw.x_arena)
    dw.close()


def test_full_7b_chain_sampled(aio):
    """The whole 7B-class chained step (32 layers and lm_head, M = 1) in one persistent launch."""
    from paper_2604_09752_gb300.workload import DeviceWorkload
    rng = np.random.default_rng(1)
    dw = DeviceWorkload(swl.WORKLOADS["7b-bf16"], seed=0, max_M=1, chained=True)
    dw.fill_chain(1)
    for _ in range(3):
        dw.step(1)
    assert aio.aio_decode_step_check(dw.step_handle(1)) == 0

    def rows_of(p):
        return np.array(sorted({0, p.N - 1, 15, 16} | set(rng.choice(p.N, 24, replace=False).tolist())))
    teacher_forced(dw, 1, "7b chain", rows_of)
    dw.close()


def test_chained_step_rejects_bad_preparations(aio):
    h = aio.aio_linear_create(11008, 64, aio.AIO_W_BF16, 2, 0)
    h2 = aio.aio_linear_create(256, 64, aio.AIO_W_BF16, 2, 0)
    h8 = aio.aio_linear_create(256, 64, aio.AIO_W_BF16, 8, 0)
    buf = torch.zeros(1 << 22, dtype=torch.uint8, device="cuda")
    p = buf.data_ptr()
    proj = [(h, p, p + (1 << 21), None, p + 65536)]
    proj2 = [(h2, p, p + (1 << 21), None, p + 65536)]
    proj8 = [(h8, p, p + (1 << 21), None, p + 65536)]
    cases = [
        # a SwiGLU x too large to stage gets a grid-wide phase of its own; a norm that large is refused
        (proj, [(aio.AIO_X_SWIGLU, p + 4096, 2 * 11008, 0, None, None, None, 0.0)], 2, 0),
        (proj, [(aio.AIO_X_RMSNORM, None, 0, 0, p + 8192, None, p, 1e-5)], 2, aio.AIO_ERR_UNSUPPORTED),
        (proj2, [(9, p + 4096, 512, 0, None, None, None, 0.0)], 1, aio.AIO_ERR_INVALID_ARG),
        (proj2, [(aio.AIO_X_SLICE, None, 512, 0, None, None, None, 0.0)], 1, aio.AIO_ERR_INVALID_ARG),
        (proj2, [(aio.AIO_X_SLICE, p + 4096, 512, 300, None, None, None, 0.0)], 1, aio.AIO_ERR_INVALID_ARG),
        (proj2, [(aio.AIO_X_SLICE, p + 4096, 512, 2, None, None, None, 0.0)], 1, aio.AIO_ERR_ALIGNMENT),
        (proj2, [(aio.AIO_X_SWIGLU, p + 4096, 300, 0, None, None, None, 0.0)], 1, aio.AIO_ERR_INVALID_ARG),
        (proj2, [(aio.AIO_X_RMSNORM, None, 0, 0, None, None, p, 1e-5)], 1, aio.AIO_ERR_INVALID_ARG),
        (proj2, [(aio.AIO_X_RMSNORM, None, 0, 0, p + 8192, p + 8192, p, 1e-5)], 1, aio.AIO_ERR_INVALID_ARG),
        (proj2, [(aio.AIO_X_RMSNORM, None, 0, 0, p + 8192, None, p, -1.0)], 1, aio.AIO_ERR_INVALID_ARG),
        (proj2, [(aio.AIO_X_RMSNORM, None, 0, 0, p + 8200, None, p, 1e-5)], 1, aio.AIO_ERR_ALIGNMENT),
        (proj8, [(aio.AIO_X_RMSNORM, None, 0, 0, p + 8192, None, p, 1e-5)], 5, aio.AIO_ERR_UNSUPPORTED),
        # attention: K = 256 is 2 heads of 128
        (proj2, [(aio.AIO_X_ATTENTION, p + 4096, 768, 0, None, None, None, 0.0, p + 8192, p + 64, 2, 64)], 1, 0),
        (proj2, [(aio.AIO_X_ATTENTION, p + 4096, 768, 0, None, None, None, 0.0, p + 8192, p + 64, 3, 64)], 1,
         aio.AIO_ERR_INVALID_ARG),                                                    # K != 128 n_heads
        (proj2, [(aio.AIO_X_ATTENTION, p + 4096, 768, 0, None, None, None, 0.0, None, p + 64, 2, 64)], 1,
         aio.AIO_ERR_INVALID_ARG),                                                    # no cache
        (proj2, [(aio.AIO_X_ATTENTION, p + 4096, 512, 0, None, None, None, 0.0, p + 8192, p + 64, 2, 64)], 1,
         aio.AIO_ERR_INVALID_ARG),                                                    # src_stride < 3K
        (proj2, [(aio.AIO_X_ATTENTION, p + 4096, 768, 0, None, None, None, 0.0, p + 8200, p + 64, 2, 64)], 1,
         aio.AIO_ERR_ALIGNMENT),                                                      # cache not 16-byte aligned
        (proj2, [(aio.AIO_X_ATTENTION, p + 4096, 768, 0, None, None, None, 0.0, p + 8192, p + 66, 2, 64)], 1,
         aio.AIO_ERR_ALIGNMENT),                                                      # L_past not 4-byte aligned
        (proj2, [(aio.AIO_X_ATTENTION, p + 4096, 768, 0, None, None, None, 0.0, p + 8192, p + 64, 2, 1)], 2,
         aio.AIO_ERR_INVALID_ARG),                                                    # L_max < M
    ]
    for pr, prep, M, status in cases:
        if status == 0:   # a valid preparation: created (not run)
            aio.aio_decode_step_destroy(aio.aio_decode_step_create_chained(pr, prep, M))
            continue
        with pytest.raises(aio.AioError) as e:
            aio.aio_decode_step_create_chained(pr, prep, M)
        assert e.value.status == status, (prep, e.value)
    aio.aio_linear_destroy(h)
    aio.aio_linear_destroy(h2)
    aio.aio_linear_destroy(h8)
