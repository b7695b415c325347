"""GPU parity of whole decode steps (every projection of every layer, Sec. 3.1), captured as one
CUDA graph with programmatic dependent launch, and of the stream-order guarantee between
consecutive projections."""
import numpy as np
import pytest
import torch

import parity
from synth import workloads as swl

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def aio():
    from paper_2604_09752_gb300 import aio as mod
    assert torch.cuda.is_available()
    return mod


def small_decoder(name, layers=2):
    wl = swl.WORKLOADS[name]
    L = max(p.layer for p in wl.projs)
    return [p for p in wl.projs if p.layer < layers or p.layer == L]


def check_workload(dw, M, what):
    for i, b in enumerate(dw.bufs):
        p = b.proj
        x = swl.gen_x(dw.seed, dw.wl, p, M).reshape(M, p.K)
        if dw.i8:
            W = swl.gen_codes(dw.seed, dw.wl, p).reshape(p.N, p.K)
            s = swl.gen_scales(dw.seed, dw.wl, p)
        else:
            W = swl.gen_w_bf16(dw.seed, dw.wl, p).reshape(p.N, p.K)
            s = None
        y_ref, mag = parity.reference(x, W, s)
        parity.check(dw.y(i, M).cpu().numpy(), y_ref, mag, p.K, f"{what} {p.name}")


@pytest.mark.parametrize("name", ["1b-bf16", "7b-int8"])
@pytest.mark.parametrize("M", [1, 3, 4, 8])
def test_small_step_graph_pdl(aio, name, M):
    from paper_2604_09752_gb300.workload import DeviceWorkload
    dw = DeviceWorkload(swl.WORKLOADS[name], seed=1, max_M=8, projs=small_decoder(name))
    dw.fill_x(M)
    dw.step(M)
    assert aio.aio_decode_step_kernels(dw.step_handle(M)) == 1            # persistent: one launch
    assert aio.aio_decode_step_kernels(dw.step_handle(M, aio.AIO_STEP_PDL)) == len(dw.bufs)
    assert aio.aio_decode_step_check(dw.step_handle(M)) == 0
    check_workload(dw, M, f"{name} M={M}")
    dw.close()


def test_step_from_host_buffers(aio):
    """aio_decode_step_host: x copied in from pinned host memory, the step, y copied back, in stream
    order; the host y equals the device y, and both meet the bar against the oracle."""
    from paper_2604_09752_gb300.workload import DeviceWorkload
    dw = DeviceWorkload(swl.WORKLOADS["7b-int8"], seed=6, max_M=2, projs=small_decoder("7b-int8", 1))
    x_host = dw.fill_x(2)
    dw.x_arena.zero_()
    dw.y_arena.fill_(0xFF)
    y_host = torch.full((dw.y_arena.numel(),), 0xAB, dtype=torch.uint8).pin_memory()
    s = torch.cuda.current_stream().cuda_stream
    aio.aio_decode_step_host(dw.step_handle(2), x_host.data_ptr(), dw.x_arena.data_ptr(), x_host.numel(),
                             dw.y_arena.data_ptr(), y_host.data_ptr(), y_host.numel(), s)
    torch.cuda.synchronize()
    assert aio.aio_decode_step_check(dw.step_handle(2)) == 0
    assert torch.equal(y_host, dw.y_arena.cpu())
    check_workload(dw, 2, "from host buffers")
    with pytest.raises(aio.AioError) as e:
        aio.aio_decode_step_host(dw.step_handle(2), None, dw.x_arena.data_ptr(), 16, 0, 0, 0, s)
    assert e.value.status == aio.AIO_ERR_INVALID_ARG
    dw.close()


@pytest.mark.parametrize("flags", [0, 1, 2, 3, 4, 5, 7])
def test_step_flag_variants_agree(aio, flags):
    from paper_2604_09752_gb300.workload import DeviceWorkload
    dw = DeviceWorkload(swl.WORKLOADS["1b-bf16"], seed=2, max_M=2, projs=small_decoder("1b-bf16", 1))
    dw.fill_x(2)
    dw.step(2, flags)
    torch.cuda.synchronize()
    ref = dw.y_arena.clone()
    dw.y_arena.zero_()
    dw.step(2, flags)
    dw.step(2, flags)
    torch.cuda.synchronize()
    assert torch.equal(ref, dw.y_arena), "steps are not bit-reproducible"
    check_workload(dw, 2, f"flags={flags}")
    dw.close()


def test_step_reads_x_only_after_previous_projection(aio):
    """Projection B's x aliases projection A's y.  A's outputs are small exact integers, so their
    fp32 bits are known on the host and B's expected input is exact; if B read x before A finished
    (a broken PDL wait), it would see the garbage written before each step."""
    rng = np.random.default_rng(0)
    KA, NA = 32768, 1024
    KB, NB = 2 * NA, 4096
    xa = np.zeros((1, KA), np.int64)
    xa[0, rng.choice(KA, 100, replace=False)] = rng.choice([-1, 1], 100)
    wa = rng.integers(-1, 2, size=(NA, KA))
    to_bf16 = {-1: 0xBF80, 0: 0, 1: 0x3F80}
    xa_b = np.vectorize(to_bf16.get, otypes=[np.uint16])(xa)
    wa_b = np.vectorize(to_bf16.get, otypes=[np.uint16])(wa)
    ya = (xa @ wa.T).astype(np.float32)                    # exact integers, |y| <= 100
    xb = ya.view(np.uint16).reshape(1, KB)                 # B's input as bf16 halves of A's fp32 output
    assert np.all(xb[0, 0::2] == 0)
    import synth
    wb = synth.normal_bf16(synth.key(99), 1.0 / np.sqrt(KB), NB * KB).reshape(NB, KB)

    def dev(a):
        return torch.from_numpy(np.ascontiguousarray(a).view(np.uint8).reshape(-1)).cuda()

    ha = aio.aio_linear_create(KA, NA, aio.AIO_W_BF16, 1, 0)
    hb = aio.aio_linear_create(KB, NB, aio.AIO_W_BF16, 1, 0)
    WA, WB = torch.empty(NA * KA * 2, dtype=torch.uint8, device="cuda"), torch.empty(NB * KB * 2, dtype=torch.uint8, device="cuda")
    aio.aio_linear_pack(ha, dev(wa_b).data_ptr(), None, WA.data_ptr(), None, 0)
    aio.aio_linear_pack(hb, dev(wb).data_ptr(), None, WB.data_ptr(), None, 0)
    XA = dev(xa_b)
    YA = torch.empty(NA, dtype=torch.float32, device="cuda")
    YB = torch.empty(NB, dtype=torch.float32, device="cuda")
    torch.cuda.synchronize()
    y_ref, mag = parity.reference(xb, wb)
    for flags in (aio.AIO_STEP_GRAPH | aio.AIO_STEP_PERSISTENT, aio.AIO_STEP_GRAPH | aio.AIO_STEP_PDL):
        step = aio.aio_decode_step_create([(ha, XA.data_ptr(), WA.data_ptr(), None, YA.data_ptr()),
                                           (hb, YA.data_ptr(), WB.data_ptr(), None, YB.data_ptr())], 1, flags)
        for it in range(5):
            YA.view(torch.int32).fill_(0x7F7F7F7F)   # garbage: huge finite bf16 halves
            YB.zero_()
            aio.aio_decode_step(step, torch.cuda.current_stream().cuda_stream)
            torch.cuda.synchronize()
            assert np.array_equal(YA.cpu().numpy(), ya[0]), "projection A wrong"
            parity.check(YB.cpu().numpy().reshape(1, NB), y_ref, mag, KB, f"flags={flags} iteration {it}")
        assert aio.aio_decode_step_check(step) == 0
        aio.aio_decode_step_destroy(step)
    aio.aio_linear_destroy(ha)
    aio.aio_linear_destroy(hb)


def test_step_rejects_bad_projection(aio):
    h = aio.aio_linear_create(256, 64, aio.AIO_W_BF16, 2, 0)
    buf = torch.zeros(1 << 20, dtype=torch.uint8, device="cuda")
    p = buf.data_ptr()
    with pytest.raises(aio.AioError) as e:
        aio.aio_decode_step_create([(h, p, p + 4096, None, p + 65536)], 3)       # M > max_M
    assert e.value.status == aio.AIO_ERR_INVALID_ARG
    with pytest.raises(aio.AioError) as e:
        aio.aio_decode_step_create([(h, p + 8, p + 4096, None, p + 65536)], 1)   # misaligned x
    assert e.value.status == aio.AIO_ERR_ALIGNMENT
    with pytest.raises(aio.AioError) as e:
        aio.aio_decode_step_create([(h, p, p + 4096, None, p + 65536)], 1, 0x40)
    assert e.value.status == aio.AIO_ERR_INVALID_ARG
    aio.aio_linear_destroy(h)
