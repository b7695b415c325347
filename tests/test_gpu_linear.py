"""GPU parity of one linear layer through the C ABI: y = x W^T (Sec. 2.1), int8 with per-channel
scales (Sec. 2.4), every width M = 1..8 the API accepts (Sec. 4.2 verification rows), packed and
row-major weights, ragged shapes, and the int8 code -128 (outside the symmetric range the recipe
draws, but a valid code the kernel must convert exactly).  Both launches of aio_linear_run are
covered: the small-projection launch (one CTA per row group) that small packed shapes take by
default, and the stream kernel (every other shape, and any handle with AIO_FLAG_STREAM_KERNEL)."""
import numpy as np
import pytest
import torch

import oracle
import parity
import synth
from oracle import layout

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def aio():
    from paper_2604_09752_gb300 import aio as mod
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    return mod


def make_inputs(K, N, M, wt, tag=0):
    x = synth.normal_bf16(synth.key(tag, K, N, 1), 1.0, M * K).reshape(M, K)
    if wt == "bf16":
        W = synth.normal_bf16(synth.key(tag, K, N, 2), 1.0 / np.sqrt(K), N * K).reshape(N, K)
        return x, W, None
    q = synth.codes_i8(synth.key(tag, K, N, 3), N * K).reshape(N, K)
    s = synth.uniform_bf16(synth.key(tag, K, N, 4), 1e-3, 1e-2, N)
    return x, q, s


def dev(a: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(a).view(np.uint8).reshape(-1)).cuda()


class Linear:
    """One handle plus device copies of its weights (packed through the C ABI unless row-major)."""

    def __init__(self, aio, W, s, max_M, rowmajor=False, flags=0):
        self.aio = aio
        self.N, self.K = W.shape
        self.i8 = W.dtype == np.int8
        wt = aio.AIO_W_INT8_PERCHANNEL if self.i8 else aio.AIO_W_BF16
        self.h = aio.aio_linear_create(self.K, self.N, wt, max_M, flags | (aio.AIO_FLAG_ROWMAJOR if rowmajor else 0))
        raw = dev(W)
        self.s = dev(s) if self.i8 else None
        if rowmajor:
            self.W = raw
        else:
            self.W = torch.empty_like(raw)
            sp = self.s.data_ptr() if self.i8 else None
            aio.aio_linear_pack(self.h, raw.data_ptr(), sp, self.W.data_ptr(), sp, 0)
        torch.cuda.synchronize()

    def run(self, x_dev, M, y_dev, stream=0):
        self.aio.aio_linear_run(self.h, x_dev.data_ptr(), M, self.K, self.N, self.W.data_ptr(),
                                self.s.data_ptr() if self.i8 else None, y_dev.data_ptr(), stream)

    def close(self):
        self.aio.aio_linear_destroy(self.h)


def n_sms():
    return torch.cuda.get_device_properties(0).multi_processor_count


def small_grid(K, N, wt):
    """The grid of the small-projection launch (one CTA per row group), or None if the shape does
    not qualify: at most 2 x SMs row groups and at most 96 KB of weights per CTA (8 warps, each
    ceil(NKT / 8) tiles of 8 KB bf16 or 4 KB int8)."""
    NG, NKT = -(-N // 16), -(-K // 256)
    tile = 4096 if wt == "int8" else 8192
    return NG if NG <= 2 * n_sms() and 8 * -(-NKT // 8) * tile <= 96 * 1024 else None


SHAPES = [(16, 1), (48, 13), (272, 9), (1040, 37), (2048, 2048), (4096, 100), (5632, 24), (11008, 40), (11008, 64)]


@pytest.mark.parametrize("wt", ["bf16", "int8"])
@pytest.mark.parametrize("K,N", SHAPES)
@pytest.mark.parametrize("M", [1, 2, 3, 4, 5, 6, 7, 8])
@pytest.mark.parametrize("layout_", ["packed", "packed-stream", "rowmajor"])
def test_linear_parity(aio, wt, K, N, M, layout_):
    x, W, s = make_inputs(K, N, M, wt)
    lin = Linear(aio, W, s, max_M=8, rowmajor=(layout_ == "rowmajor"),
                 flags=aio.AIO_FLAG_STREAM_KERNEL if layout_ == "packed-stream" else 0)
    grid = aio.aio_linear_launch_info(lin.h)["grid"]
    want = small_grid(K, N, wt) if layout_ == "packed" else None   # None: the stream kernel, one CTA per SM
    assert grid == (want if want is not None else n_sms()), (grid, want)
    xd = dev(x)
    guard = 64
    yd = torch.full((M * N + 2 * guard,), 12345.0, dtype=torch.float32, device="cuda")
    ypart = yd[guard: guard + M * N]
    lin.run(xd, M, ypart)
    torch.cuda.synchronize()
    assert aio.aio_linear_check(lin.h) == 0
    out = yd.cpu().numpy()
    assert np.all(out[:guard] == 12345.0) and np.all(out[guard + M * N:] == 12345.0), "guard band overwritten"
    y_ref, mag = parity.reference(x, W, s)
    parity.check(out[guard: guard + M * N].reshape(M, N), y_ref, mag, K, f"{wt} K={K} N={N} M={M} {layout_}")
    lin.close()


@pytest.mark.parametrize("wt,K", [("bf16", 2048), ("bf16", 2064), ("int8", 6144), ("int8", 6160)])
@pytest.mark.parametrize("N", [4864, 4865])
def test_small_launch_limits(aio, wt, K, N):
    """At and just past the small-projection launch's limits: 2 x 152 row groups (N = 4864) and
    96 KB of weights per CTA (bf16 K = 2048, int8 K = 6144, one tile per warp more past them).
    Inside, one CTA per row group; outside, the stream kernel; both meet the bar at M = 8."""
    M = 8
    x, W, s = make_inputs(K, N, M, wt, tag=13)
    lin = Linear(aio, W, s, max_M=8)
    want = small_grid(K, N, wt)
    inside = N == 4864 and K in (2048, 6144)
    assert (want is not None) == inside
    assert aio.aio_linear_launch_info(lin.h)["grid"] == (want if inside else n_sms())
    y = torch.full((M * N,), float("nan"), dtype=torch.float32, device="cuda")
    lin.run(dev(x), M, y)
    torch.cuda.synchronize()
    assert aio.aio_linear_check(lin.h) == 0
    y_ref, mag = parity.reference(x, W, s)
    parity.check(y.cpu().numpy().reshape(M, N), y_ref, mag, K, f"limits {wt} K={K} N={N}")
    lin.close()


@pytest.mark.parametrize("wt", ["bf16", "int8"])
@pytest.mark.parametrize("K,N", [(16, 1), (272, 9), (1040, 37), (4096, 20), (11008, 17)])
def test_pack_matches_oracle_layout_and_unpacks(aio, wt, K, N):
    x, W, s = make_inputs(K, N, 1, wt, tag=7)
    lin = Linear(aio, W, s, max_M=1)
    packed = lin.W.cpu().numpy().view(W.dtype)
    assert np.array_equal(packed, layout.pack_tiles(W)), "packer differs from the layout definition"
    back = torch.empty_like(lin.W)
    aio.aio_linear_unpack(lin.h, lin.W.data_ptr(), back.data_ptr(), 0)
    torch.cuda.synchronize()
    assert np.array_equal(back.cpu().numpy().view(W.dtype).reshape(N, K), W)
    if wt == "int8":
        assert np.array_equal(lin.s.cpu().numpy().view(np.uint16), s)
    lin.close()


def test_one_hot_x_selects_weight_column(aio):
    K, N = 1040, 300
    _, W, _ = make_inputs(K, N, 1, "bf16", tag=3)
    lin = Linear(aio, W, None, max_M=8)
    ks = [0, 1, 255, 256, 257, 1039]
    x = np.zeros((len(ks), K), np.uint16)
    for m, k in enumerate(ks):
        x[m, k] = 0x3F80  # 1.0
    y = torch.empty(len(ks) * N, dtype=torch.float32, device="cuda")
    lin.run(dev(x), len(ks), y)
    torch.cuda.synchronize()
    got = y.cpu().numpy().reshape(len(ks), N)
    want = (W[:, ks].T.astype(np.uint32) << 16).view(np.float32)
    assert np.array_equal(got, want)
    lin.close()


def test_int8_known_codes_exact(aio):
    # one-hot x: y = s * q exactly; 2^-7 * -127 = -0.9921875 and bf16(0.005) * 127 = 0.6356201171875
    K, N = 16, 2
    q = np.zeros((N, K), np.int8)
    q[0, 3], q[1, 3] = -127, 127
    s = np.array([0x3C00, 0x3BA4], np.uint16)
    x = np.zeros((1, K), np.uint16)
    x[0, 3] = 0x3F80
    lin = Linear(aio, q, s, max_M=1)
    y = torch.empty(N, dtype=torch.float32, device="cuda")
    lin.run(dev(x), 1, y)
    torch.cuda.synchronize()
    assert y.cpu().numpy().tolist() == [-0.9921875, np.float32(0.0050048828125 * 127)]
    lin.close()


@pytest.mark.parametrize("K,N,layout_", [(16, 3, "packed"), (4096, 64, "packed"), (1040, 37, "packed"),
                                         (4096, 64, "rowmajor")])
def test_int8_code_minus_128_one_hot_exact(aio, K, N, layout_):
    """q = -128 in the columns the one-hot x rows select (full, ragged and row-major tiles), a few bf16
    scales: y[m, n] = s[n] * -128 exactly (s * 2^7 is exact in fp32 and in the oracle's double)."""
    ks = [0, 1, 255, 256, K - 1] if K > 256 else [0, 3, K - 1]
    q = synth.codes_i8(synth.key(21, K, N), N * K).reshape(N, K)
    q[:, ks] = -128
    # a few bf16 scales: 2^-7, bf16(0.005), the smallest and largest of the recipe's range
    s = np.resize(np.array([0x3C00, 0x3BA4, 0x3A83, 0x3C24], np.uint16), N)
    x = np.zeros((len(ks), K), np.uint16)
    for m, k in enumerate(ks):
        x[m, k] = 0x3F80
    lin = Linear(aio, q, s, max_M=8, rowmajor=(layout_ == "rowmajor"))
    y = torch.empty(len(ks) * N, dtype=torch.float32, device="cuda")
    lin.run(dev(x), len(ks), y)
    torch.cuda.synchronize()
    got = y.cpu().numpy().reshape(len(ks), N)
    want = (s.astype(np.uint32) << 16).view(np.float32) * np.float32(-128.0)
    assert np.array_equal(got, np.broadcast_to(want, got.shape))
    y_ref, _ = parity.reference(x, q, s)
    assert np.array_equal(got.astype(np.float64), y_ref)
    lin.close()


@pytest.mark.parametrize("K,N", [(4096, 64), (1040, 37), (11008, 40)])
@pytest.mark.parametrize("M", [1, 4, 8])
def test_int8_rows_of_minus_128_and_full_code_range(aio, K, N, M):
    """Whole rows of -128 (every second row group's first row, and the last row) inside weights that
    take every int8 code in [-128, 127], against the fp64 oracle at the stated bar."""
    x, _, s = make_inputs(K, N, M, "int8", tag=23)
    u = synth.codes_i8(synth.key(23, K, N, 9), N * K).astype(np.int16).reshape(N, K)
    # every int8 code: 127 stays at odd k and becomes -128 at even k
    q = np.where((u == 127) & (np.arange(K) % 2 == 0), -128, u).astype(np.int8)
    q[0::32] = -128
    q[N - 1] = -128
    assert (q == -128).any(axis=1).sum() >= 2 and (q == -128).sum() > N
    for rowmajor in (False, True):
        lin = Linear(aio, q, s, max_M=8, rowmajor=rowmajor)
        y = torch.full((M * N,), float("nan"), dtype=torch.float32, device="cuda")
        lin.run(dev(x), M, y)
        torch.cuda.synchronize()
        assert aio.aio_linear_check(lin.h) == 0
        y_ref, mag = parity.reference(x, q, s)
        parity.check(y.cpu().numpy().reshape(M, N), y_ref, mag, K, f"-128 K={K} N={N} M={M} rowmajor={rowmajor}")
        lin.close()


def test_deterministic_and_repeatable(aio):
    x, W, _ = make_inputs(4096, 4096, 2, "bf16", tag=5)
    lin = Linear(aio, W, None, max_M=2)
    xd = dev(x)
    y1 = torch.empty(2 * 4096, dtype=torch.float32, device="cuda")
    y2 = torch.empty_like(y1)
    lin.run(xd, 2, y1)
    for _ in range(3):
        lin.run(xd, 2, y2)
    torch.cuda.synchronize()
    assert torch.equal(y1.view(torch.int32), y2.view(torch.int32))
    lin.close()


def test_argument_errors_launch_nothing(aio):
    x, W, s = make_inputs(256, 64, 1, "int8", tag=9)
    lin = Linear(aio, W, s, max_M=2)
    xd = dev(x)
    y = torch.full((64,), 7.0, dtype=torch.float32, device="cuda")
    K, N = 256, 64
    cases = [
        (dict(M=3), aio.AIO_ERR_INVALID_ARG),                     # M > max_M
        (dict(M=0), aio.AIO_ERR_INVALID_ARG),
        (dict(K=272), aio.AIO_ERR_INVALID_ARG),                   # shape mismatch
        (dict(N=65), aio.AIO_ERR_INVALID_ARG),
        (dict(scales=None), aio.AIO_ERR_INVALID_ARG),             # int8 without scales
        (dict(x=xd.data_ptr() + 8), aio.AIO_ERR_ALIGNMENT),       # misaligned x
        (dict(y=y.data_ptr() + 4), aio.AIO_ERR_ALIGNMENT),
        (dict(W=lin.W.data_ptr() + 2), aio.AIO_ERR_ALIGNMENT),
        (dict(scales=lin.s.data_ptr() + 1), aio.AIO_ERR_ALIGNMENT),
        (dict(x=None), aio.AIO_ERR_INVALID_ARG),
    ]
    for over, code in cases:
        args = dict(h=lin.h, x=xd.data_ptr(), M=1, K=K, N=N, W=lin.W.data_ptr(), scales=lin.s.data_ptr(),
                    y=y.data_ptr(), stream=0)
        args.update(over)
        with pytest.raises(aio.AioError) as e:
            aio.aio_linear_run(**args)
        assert e.value.status == code, (over, e.value)
    torch.cuda.synchronize()
    assert torch.all(y == 7.0), "a rejected call launched work"
    # bf16 handle given scales
    x2, W2, _ = make_inputs(256, 64, 1, "bf16", tag=9)
    lin2 = Linear(aio, W2, None, max_M=1)
    with pytest.raises(aio.AioError) as e:
        aio.aio_linear_run(lin2.h, xd.data_ptr(), 1, K, N, lin2.W.data_ptr(), lin.s.data_ptr(), y.data_ptr(), 0)
    assert e.value.status == aio.AIO_ERR_INVALID_ARG
    lin.close()
    lin2.close()


@pytest.mark.parametrize("kernel", ["small", "stream"])
def test_bounded_wait_reports_timeout_and_context_survives(aio, kernel):
    # AIO_FLAG_TEST_STALL: one warp never receives its first tile; its wait gives up after 20 ms,
    # the kernel returns, and the host reads AIO_ERR_DEVICE_TIMEOUT.  The context stays usable.
    x, W, _ = make_inputs(2048, 512, 1, "bf16", tag=11)
    extra = aio.AIO_FLAG_STREAM_KERNEL if kernel == "stream" else 0
    assert small_grid(2048, 512, "bf16") == 32
    stall = Linear(aio, W, None, max_M=1, flags=aio.AIO_FLAG_TEST_STALL | extra)
    assert aio.aio_linear_launch_info(stall.h)["grid"] == (32 if kernel == "small" else n_sms())
    y = torch.empty(512, dtype=torch.float32, device="cuda")
    stall.run(dev(x), 1, y)
    with pytest.raises(aio.AioError) as e:
        aio.aio_linear_check(stall.h)
    assert e.value.status == aio.AIO_ERR_DEVICE_TIMEOUT
    aio.aio_linear_reset(stall.h)
    stall.close()
    good = Linear(aio, W, None, max_M=1)
    good.run(dev(x), 1, y)
    assert aio.aio_linear_check(good.h) == 0
    y_ref, mag = parity.reference(x, W)
    parity.check(y.cpu().numpy().reshape(1, -1), y_ref, mag, 2048, "after timeout")
    good.close()


def test_oom_injection_on_host(aio, monkeypatch):
    monkeypatch.setenv("AIO_TEST_FAIL_ALLOC", "1")
    with pytest.raises(aio.AioError) as e:
        aio.aio_linear_create(256, 64, aio.AIO_W_BF16, 1, 0)
    assert e.value.status == aio.AIO_ERR_OOM


def test_probe_reads_everything(aio):
    n = 64 << 20
    buf = torch.randint(0, 2**31 - 1, (n // 4,), dtype=torch.int32, device="cuda")
    out = torch.zeros(1, dtype=torch.int32, device="cuda")
    aio.aio_probe_read(buf.data_ptr(), n, out.data_ptr(), 0)
    torch.cuda.synchronize()
    # the probe XORs word (lane * 32) of every 4 KB chunk over the 32 lanes
    b = buf.view(-1, 1024)[:, ::32].cpu().numpy().astype(np.uint32)
    expect = np.bitwise_xor.reduce(b.ravel())
    assert np.uint32(out.item() & 0xFFFFFFFF) == expect
