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


@pytest.mark.parametrize("dtype", [np.uint16, np.int8])
def test_tiles_are_contiguous_and_ordered(dtype):
    N, K = 20, 600      # ragged row group (4 rows) and ragged k tile (88 columns)
    idx = np.arange(N * K, dtype=np.int64).reshape(N, K)
    W = (idx % 251).astype(dtype)
    assert np.array_equal(layout.unpack_tiles(layout.pack_tiles(W), N, K), W)
    Pi = _pack_index(idx, np.dtype(dtype).itemsize)
    pos = 0
    for g in range(3):
        rows = min(8, N - 8 * g)
        for kt in range(3):
            ln = min(256, K - 256 * kt)
            assert layout.tile_offset(N, K, g, kt) == pos
            blk = Pi[pos:pos + rows * ln]
            # every tile holds exactly its own block of W; ragged tiles are row-major
            assert np.array_equal(np.sort(blk), np.sort(idx[8 * g:8 * g + rows, 256 * kt:256 * kt + ln].ravel()))
            if rows < 8 or ln < 256:
                assert np.array_equal(blk.reshape(rows, ln), idx[8 * g:8 * g + rows, 256 * kt:256 * kt + ln])
            pos += rows * ln
    assert pos == N * K


def _pack_index(idx, esize):
    """The layout applied to an index matrix, with the element size of the real dtype."""
    order = layout._full_tile_order(esize)
    N, K = idx.shape
    out = np.empty(N * K, dtype=np.int64)
    for g in range((N + 7) // 8):
        rows = min(8, N - 8 * g)
        for kt in range((K + 255) // 256):
            ln = min(256, K - 256 * kt)
            blk = idx[8 * g:8 * g + rows, 256 * kt:256 * kt + ln].reshape(-1)
            if rows == 8 and ln == 256:
                blk = blk[order]
            off = layout.tile_offset(N, K, g, kt)
            out[off:off + rows * ln] = blk
    return out


@pytest.mark.parametrize("esize,P", [(2, 8), (1, 16)])
def test_full_tile_fragment_order(esize, P):
    # lane L = 4r + c reads piece j at byte j*512 + L*16: W[r, 64c + P j : 64c + P (j+1)]
    order = layout._full_tile_order(esize)
    assert np.array_equal(np.sort(order), np.arange(8 * 256))
    for j in range(256 // (4 * P)):
        for L in (0, 5, 31):
            r, c = divmod(L, 4)
            pos = (j * 512 + L * 16) // esize
            assert list(order[pos:pos + P]) == [r * 256 + 64 * c + P * j + e for e in range(P)]
