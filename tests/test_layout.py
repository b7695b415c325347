"""The tiled weight layout (oracle-side definition): a pure, padding-free permutation (CPU)."""
import numpy as np
import pytest

from oracle import layout


@pytest.mark.parametrize("N,K", [(1, 16), (8, 256), (9, 272), (17, 1040), (64, 512), (3, 4096), (13, 5632)])
@pytest.mark.parametrize("dtype", [np.uint16, np.int8])
def test_pack_unpack_roundtrip(N, K, dtype):
    rng = np.random.default_rng(N * K)
    W = rng.integers(-100, 100, size=(N, K)).astype(dtype)
    P = layout.pack_tiles(W)
    assert P.size == N * K
    assert np.array_equal(np.sort(P), np.sort(W.ravel()))
    assert np.array_equal(layout.unpack_tiles(P, N, K), W)


def test_tiles_are_contiguous_and_ordered():
    N, K = 20, 600      # ragged row group (4 rows) and ragged k tile (88 columns)
    idx = np.arange(N * K, dtype=np.int64).reshape(N, K)
    P = layout.pack_tiles(idx)
    pos = 0
    for g in range(3):
        rows = min(8, N - 8 * g)
        for kt in range(3):
            ln = min(256, K - 256 * kt)
            assert layout.tile_offset(N, K, g, kt) == pos
            blk = P[pos:pos + rows * ln].reshape(rows, ln)
            assert np.array_equal(blk, idx[8 * g:8 * g + rows, 256 * kt:256 * kt + ln])
            pos += rows * ln
    assert pos == N * K
