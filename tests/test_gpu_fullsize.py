"""GPU parity at the full 7B-class sizes, in the launch configuration bench.py times: one persistent
launch per decode step, captured in a CUDA graph, every weight of all 129 projections resident.
Each projection is checked on sampled output rows that the fp64 oracle computes one by one from
regenerated weight rows (the first and last row, the rows around the first 16-row group boundary,
the middle row, and random rows)."""
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


def sample_rows(N, rng, n=40):
    fixed = {0, N - 1, 15, 16, 17, N // 2}
    rnd = set(rng.choice(N, size=min(n, N), replace=False).tolist())
    return np.array(sorted(fixed | rnd), dtype=np.int64)


def check_sampled(dw, M, what, rng, x_of=None):
    for i, b in enumerate(dw.bufs):
        p = b.proj
        rows = sample_rows(p.N, rng)
        x = x_of(i) if x_of else swl.gen_x(dw.seed, dw.wl, p, M).reshape(M, p.K)
        Wr, Sr = swl.gen_rows(dw.seed, dw.wl, p, rows)
        y_ref, mag = parity.reference(x, Wr, Sr)
        assert bool(torch.isfinite(dw.y(i, M)).all()), f"{what} {p.name}: an output was not written"
        y = dw.y(i, M)[:, torch.from_numpy(rows).cuda()].cpu().numpy()
        parity.check(y, y_ref, mag, p.K, f"{what} {p.name}")


@pytest.mark.parametrize("name", ["7b-bf16", "7b-int8"])
def test_full_7b_step_sampled(aio, name):
    from paper_2604_09752_gb300.workload import DeviceWorkload
    rng = np.random.default_rng(0)
    dw = DeviceWorkload(swl.WORKLOADS[name], seed=0, max_M=8)
    flags = aio.AIO_STEP_GRAPH | aio.AIO_STEP_PERSISTENT
    for M in (1, 4, 8):   # M = 4 and 8 at K = 11008 read x unstaged
        dw.fill_x(M)
        dw.y_arena.fill_(0xFF)                      # NaN everywhere: every output must be written
        for _ in range(3):
            dw.step(M, flags)
        assert aio.aio_decode_step_check(dw.step_handle(M, flags)) == 0
        assert aio.aio_decode_step_kernels(dw.step_handle(M, flags)) == 1
        check_sampled(dw, M, f"{name} M={M}", rng)
    dw.close()
