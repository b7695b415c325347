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
    N, K = 40, 600      # ragged row group (8 rows) and ragged k tile (88 columns)
    R = layout.ROWS_PER_GROUP
    assert R == 16
    idx = np.arange(N * K, dtype=np.int64).reshape(N, K)
    W = (idx % 251).astype(dtype)
    assert np.array_equal(layout.unpack_tiles(layout.pack_tiles(W), N, K), W)
    Pi = _pack_index(idx, np.dtype(dtype).itemsize)
    pos = 0
    for g in range(3):
        rows = min(R, N - R * g)
        for kt in range(3):
            T = layout.K_TILE
            ln = min(T, K - T * kt)
            assert layout.tile_offset(N, K, g, kt) == pos
            blk = Pi[pos:pos + rows * ln]
            # every tile holds exactly its own block of W; ragged tiles are row-major
            assert np.array_equal(np.sort(blk), np.sort(idx[R * g:R * g + rows, T * kt:T * kt + ln].ravel()))
            if rows < R or ln < T:
                assert np.array_equal(blk.reshape(rows, ln), idx[R * g:R * g + rows, T * kt:T * kt + ln])
            pos += rows * ln
    assert pos == N * K


def _pack_index(idx, esize):
    """The layout applied to an index matrix, with the element size of the real dtype."""
    R = layout.ROWS_PER_GROUP
    order = layout._full_tile_order(esize)
    N, K = idx.shape
    out = np.empty(N * K, dtype=np.int64)
    for g in range((N + R - 1) // R):
        rows = min(R, N - R * g)
        T = layout.K_TILE
        for kt in range((K + T - 1) // T):
            ln = min(T, K - T * kt)
            blk = idx[R * g:R * g + rows, T * kt:T * kt + ln].reshape(-1)
            if rows == R and ln == T:
                blk = blk[order]
            off = layout.tile_offset(N, K, g, kt)
            out[off:off + rows * ln] = blk
    return out


def test_full_tile_fragment_order_bf16():
    # lane L = 4r + c reads piece s (16 B) at byte s*512 + 16L: one MMA A fragment for k-step s,
    # k0 = 32*(s // 2) + 8c + 4*(s % 2): W[r, k0:k0+2], W[r+8, k0:k0+2], W[r, k0+2:k0+4], W[r+8, k0+2:k0+4]
    T = layout.K_TILE
    assert T == 256
    order = layout._full_tile_order(2)
    assert np.array_equal(np.sort(order), np.arange(16 * T))
    cases = {(0, 0): (0, 0), (1, 0): (0, 4), (0, 1): (0, 8), (2, 0): (0, 32), (15, 31): (7, 224 + 24 + 4),
             (5, 6): (1, 64 + 16 + 4), (8, 13): (3, 128 + 8)}
    for (s, L), (r, k0) in cases.items():
        pos = (s * 512 + L * 16) // 2
        want = [(r, k0), (r, k0 + 1), (r + 8, k0), (r + 8, k0 + 1), (r, k0 + 2), (r, k0 + 3), (r + 8, k0 + 2),
                (r + 8, k0 + 3)]
        assert list(order[pos:pos + 8]) == [row * T + k for row, k in want], (s, L)


def test_full_tile_fragment_order_int8():
    # piece j (16 codes) of lane L = 4r + c: row r + 8*(j // 4); bytes 0-7 k = 64u + 8c, bytes 8-15 k = 64u + 32 + 8c
    T = layout.K_TILE
    order = layout._full_tile_order(1)
    assert np.array_equal(np.sort(order), np.arange(16 * T))
    cases = {(0, 0): (0, 0, 32), (1, 2): (0, 64 + 16, 64 + 32 + 16), (3, 31): (7, 192 + 24, 224 + 24),
             (4, 0): (8, 0, 32), (7, 13): (3 + 8, 192 + 8, 224 + 8)}
    for (j, L), (row, ka, kb) in cases.items():
        pos = j * 512 + L * 16
        swz = (0, 2, 1, 3, 4, 6, 5, 7)   # each 4-code word holds k pairs (0,1) in its low bytes, (2,3) in its high bytes
        want = [row * T + ka + e for e in swz] + [row * T + kb + e for e in swz]
        assert list(order[pos:pos + 16]) == want, (j, L)


@pytest.mark.parametrize("esize", [2, 1])
def test_lane_reads_cover_each_mma_k_step(esize):
    # The kernel's k-permutation: k-step s (K_TILE/16 of them) uses, in lane (g, c), k = 32(s//2) + 8c + 4(s%2)
    # + 0..3 of rows g and g + 8.  Every (row, k) of the tile is used by exactly one (lane, step), and the
    # lane's pieces hold those k.
    T = layout.K_TILE
    order = layout._full_tile_order(esize)
    per_piece = 16 // esize
    seen = np.zeros(16 * T, dtype=int)
    for L in range(32):
        g, c = divmod(L, 4)
        held = set()
        for j in range(16 * T * esize // 512):
            pos = (j * 512 + L * 16) // esize
            held.update(order[pos:pos + per_piece].tolist())
        for s in range(T // 16):
            for row in (g, g + 8):
                for e in range(4):
                    k = 32 * (s // 2) + 8 * c + 4 * (s % 2) + e
                    assert row * T + k in held
                    seen[row * T + k] += 1
    assert np.all(seen == 1)
