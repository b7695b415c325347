"""aio_linear_run_noalloc: the linear run for callers that cannot allocate device memory where they
call (an engine whose pools hold nearly all of HBM, or a loop in which cudaMalloc would synchronise
the device).  Its scratch is a static device array inside the library, and nothing is allocated.

Each case runs two calls in a row on one stream (the second reuses the scratch the first left) and
checks both against the fp64 oracle at the linear-layer bar (parity.check), and bit for bit against
aio_linear_run of a handle created with AIO_FLAG_STREAM_KERNEL on the same inputs: the launch, the
partition and the summation order are the same.

The file name sorts last so the test also runs after every other GPU test in one session."""
import numpy as np
import pytest
import torch

import parity
import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def aio():
    from paper_2604_09752_gb300 import aio as mod
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    return mod


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a).view(np.uint8).reshape(-1)).cuda()


def _inputs(K, N, M, wt):
    x = synth.normal_bf16(synth.key(41, K, N, 1), 1.0, M * K).reshape(M, K)
    if wt == "bf16":
        return x, synth.normal_bf16(synth.key(41, K, N, 2), 1.0 / np.sqrt(K), N * K).reshape(N, K), None
    q = synth.codes_i8(synth.key(41, K, N, 3), N * K).reshape(N, K)
    return x, q, synth.uniform_bf16(synth.key(41, K, N, 4), 1e-3, 1e-2, N)


def _weights(aio, W, s, K, N, M, wt_c, flags):
    """A handle (for the aio_linear_run comparison and the packer) and the device weights.  The
    handle takes the stream kernel, as the no-alloc entry does, whatever the shape."""
    h = aio.aio_linear_create(K, N, wt_c, M, flags | aio.AIO_FLAG_STREAM_KERNEL)
    raw = _dev(W)
    sd = _dev(s) if s is not None else None
    sp = sd.data_ptr() if sd is not None else None
    if flags & aio.AIO_FLAG_ROWMAJOR:
        Wd = raw
    else:
        Wd = torch.empty_like(raw)
        aio.aio_linear_pack(h, raw.data_ptr(), sp, Wd.data_ptr(), sp, 0)
    torch.cuda.synchronize()
    return h, Wd, sd, sp


@pytest.mark.parametrize("wt", ["bf16", "int8"])
@pytest.mark.parametrize("K,N,M,rowmajor", [(4096, 32000, 1, False), (11008, 4096, 8, False), (11008, 4096, 4, False),
                                            (1040, 37, 3, False), (4096, 1000, 2, True)])
def test_noalloc_matches_oracle_and_linear_run(aio, wt, K, N, M, rowmajor):
    x, W, s = _inputs(K, N, M, wt)
    wt_c = aio.AIO_W_INT8_PERCHANNEL if wt == "int8" else aio.AIO_W_BF16
    flags = aio.AIO_FLAG_ROWMAJOR if rowmajor else 0
    h, Wd, sd, sp = _weights(aio, W, s, K, N, M, wt_c, flags)
    xd = _dev(x)
    y_run = torch.empty(M * N, dtype=torch.float32, device="cuda")
    aio.aio_linear_run(h, xd.data_ptr(), M, K, N, Wd.data_ptr(), sp, y_run.data_ptr(), 0)
    y1 = torch.full((M * N,), float("nan"), dtype=torch.float32, device="cuda")
    y2 = torch.full_like(y1, float("nan"))
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    stream = torch.cuda.current_stream().cuda_stream
    # a first call does the per-device set-up (which may load the library image's static scratch)
    aio.aio_linear_run_noalloc(xd.data_ptr(), M, K, N, wt_c, flags, Wd.data_ptr(), sp, y1.data_ptr(),
                               err.data_ptr(), stream)
    y1.fill_(float("nan"))
    torch.cuda.synchronize()
    assert aio.aio_linear_check(h) == 0
    free0 = torch.cuda.mem_get_info()[0]
    for y in (y1, y2):   # back to back on one stream: the second reuses the scratch the first left
        aio.aio_linear_run_noalloc(xd.data_ptr(), M, K, N, wt_c, flags, Wd.data_ptr(), sp, y.data_ptr(),
                                   err.data_ptr(), stream)
    torch.cuda.synchronize()
    assert err.item() == 0, "a bounded device wait expired"
    assert torch.cuda.mem_get_info()[0] == free0, "device memory was allocated"
    y_ref, mag = parity.reference(x, W, s)
    for i, y in enumerate((y1, y2)):
        assert torch.isfinite(y).all(), f"call {i + 1}: output not fully written"
        parity.check(y.cpu().numpy().reshape(M, N), y_ref, mag, K, f"noalloc call {i + 1} {wt} K={K} N={N} M={M}")
        assert torch.equal(y.view(torch.int32), y_run.view(torch.int32)), f"call {i + 1}: differs from aio_linear_run"
    aio.aio_linear_destroy(h)


def test_noalloc_error_word_is_sticky_and_scratch_recovers(aio):
    """A non-zero device_error (left by an earlier failed call) is never cleared by the library, and
    the call that sees it gives up its waits for other warps' partial sums; once the caller clears
    the word, the next call is correct again (each call empties the scratch slots it uses)."""
    K, N, M = 11008, 4096, 2          # row groups split between warps: owners gather partial sums
    x, W, s = _inputs(K, N, M, "bf16")
    h, Wd, _, _ = _weights(aio, W, s, K, N, M, aio.AIO_W_BF16, 0)
    xd = _dev(x)
    y = torch.full((M * N,), float("nan"), dtype=torch.float32, device="cuda")
    err = torch.full((1,), 5, dtype=torch.int32, device="cuda")
    stream = torch.cuda.current_stream().cuda_stream
    aio.aio_linear_run_noalloc(xd.data_ptr(), M, K, N, aio.AIO_W_BF16, 0, Wd.data_ptr(), None, y.data_ptr(),
                               err.data_ptr(), stream)
    torch.cuda.synchronize()
    assert err.item() == 5, "the library changed a caller-owned error word"
    err.zero_()
    y.fill_(float("nan"))
    aio.aio_linear_run_noalloc(xd.data_ptr(), M, K, N, aio.AIO_W_BF16, 0, Wd.data_ptr(), None, y.data_ptr(),
                               err.data_ptr(), stream)
    torch.cuda.synchronize()
    assert err.item() == 0
    y_ref, mag = parity.reference(x, W, s)
    parity.check(y.cpu().numpy().reshape(M, N), y_ref, mag, K, "after a cleared error word")
    aio.aio_linear_destroy(h)


def test_noalloc_rejects_oversize_and_bad_arguments(aio, monkeypatch):
    K, N = 256, 64
    x, W, _ = _inputs(K, N, 1, "bf16")
    xd, Wd = _dev(x), _dev(W)
    y = torch.full((N,), 7.0, dtype=torch.float32, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    bf = aio.AIO_W_BF16
    base = dict(x=xd.data_ptr(), M=1, K=K, N=N, wt=bf, flags=0, W=Wd.data_ptr(), scales=None,
                y=y.data_ptr(), device_error=err.data_ptr(), stream=0)
    cases = [
        (dict(M=9), aio.AIO_ERR_INVALID_ARG, None),
        (dict(K=17), aio.AIO_ERR_INVALID_ARG, None),
        (dict(device_error=None), aio.AIO_ERR_INVALID_ARG, None),
        (dict(device_error=err.data_ptr() + 2), aio.AIO_ERR_ALIGNMENT, None),
        (dict(flags=aio.AIO_FLAG_TEST_STALL), aio.AIO_ERR_INVALID_ARG, None),
        (dict(wt=aio.AIO_W_INT8_PERCHANNEL), aio.AIO_ERR_INVALID_ARG, None),   # int8 without scales
        (dict(x=xd.data_ptr() + 8), aio.AIO_ERR_ALIGNMENT, None),
    ]
    for over, code, word in cases:
        args = dict(base)
        args.update(over)
        with pytest.raises(aio.AioError) as e:
            aio.aio_linear_run_noalloc(**args)
        assert e.value.status == code, (over, str(e.value))
        if word:
            assert word in str(e.value)
    # beyond the static scratch: every M <= 8 fits a GB300's 1 MiB, so the test lowers the limit
    monkeypatch.setenv("AIO_TEST_NOALLOC_BYTES", "4096")
    with pytest.raises(aio.AioError) as e:
        aio.aio_linear_run_noalloc(**base)
    assert e.value.status == aio.AIO_ERR_INVALID_ARG and "scratch" in str(e.value)
    monkeypatch.delenv("AIO_TEST_NOALLOC_BYTES")
    torch.cuda.synchronize()
    assert torch.all(y == 7.0), "a rejected call launched work"
    assert err.item() == 0
