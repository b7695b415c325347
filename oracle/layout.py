"""Reference definition of the tiled weight layout (TEST INFRASTRUCTURE).

The CUDA packer reorders W [N, K] (bf16 or int8) into tiles so that each streamed run of tiles
is one contiguous block of bytes, and so that a full tile sits in shared memory in the order the
kernel's lanes read it.  The layout is a pure permutation of the elements, written here with
plain numpy slicing so the GPU packer can be checked bit for bit against it:

  * rows are grouped 16 at a time: row group g holds rows [16g, 16g + rows_g),
    rows_g = min(16, N - 16g); the group starts at element offset 16 g K;
  * inside a group, k is cut into tiles of 256 columns: tile kt covers
    [256 kt, 256 kt + len_kt), len_kt = min(256, K - 256 kt), and starts at
    element offset rows_g * 256 * kt from the start of its group;
  * a full tile (rows_g = 16, len_kt = 256) is stored as 16-byte pieces, 32 lanes per piece
    index: lane L = 4 r + c (r = 0..7, c = 0..3) reads piece j at byte j * 512 + 16 L of the
    tile:
      - 2-byte elements: piece s (0..15) holds, with k0 = 32 (s // 2) + 8 c + 4 (s % 2), the
        pairs W[r, k0:k0+2], W[r+8, k0:k0+2], W[r, k0+2:k0+4], W[r+8, k0+2:k0+4] (one MMA's A
        fragment, in register order);
      - 1-byte elements: pieces hold runs of 8 consecutive k, W[row, 32 t + 8 c : 32 t + 8 c + 8];
        piece j (0..7) is row r + 8 (j // 4), runs t = 2 (j % 4) then
        2 (j % 4) + 1 (8 bytes each), each run stored as k + (0, 2, 1, 3, 4, 6, 5, 7): in every
        4-byte word the codes of the first k pair sit in the low bytes of the two 16-bit halves
        and those of the second pair in the high bytes;
  * a ragged tile is the row-major block [rows_g, len_kt].

No padding is added, so the packed buffer has exactly N*K elements.
"""
from __future__ import annotations

import numpy as np

ROWS_PER_GROUP = 16
K_TILE = 256
INT8_RUN_ORDER = np.array([0, 2, 1, 3, 4, 6, 5, 7])   # storage order of an 8-code run in a full int8 tile


def tile_offset(N: int, K: int, g: int, kt: int) -> int:
    rows_g = min(ROWS_PER_GROUP, N - ROWS_PER_GROUP * g)
    return ROWS_PER_GROUP * g * K + rows_g * K_TILE * kt


def _lane_runs(esize: int, j: int, L: int):
    """int8: the (row, first k) of the 8-code runs that piece j of lane L holds, in storage order."""
    r, c = divmod(L, 4)
    per_half = K_TILE // 64
    u = j % per_half
    row = r + 8 * (j // per_half)
    return [(row, 32 * (2 * u) + 8 * c), (row, 32 * (2 * u + 1) + 8 * c)]


def _bf16_piece(s: int, L: int):
    """(row, k) of the 8 elements of bf16 piece s of lane L, in storage order."""
    r, c = divmod(L, 4)
    k0 = 32 * (s // 2) + 8 * c + 4 * (s % 2)
    return [(r, k0), (r, k0 + 1), (r + 8, k0), (r + 8, k0 + 1),
            (r, k0 + 2), (r, k0 + 3), (r + 8, k0 + 2), (r + 8, k0 + 3)]


def _full_tile_order(esize: int) -> np.ndarray:
    """order[i] = row-major index (r * 256 + k) of the element stored at position i of a full tile."""
    pieces = ROWS_PER_GROUP * K_TILE * esize // 512      # 16-byte pieces per lane
    order = np.empty(ROWS_PER_GROUP * K_TILE, dtype=np.int64)
    for j in range(pieces):
        for L in range(32):
            pos = (j * 512 + L * 16) // esize
            if esize == 2:
                order[pos:pos + 8] = [row * K_TILE + k for row, k in _bf16_piece(j, L)]
                continue
            for row, k0 in _lane_runs(esize, j, L):
                order[pos:pos + 8] = row * K_TILE + k0 + INT8_RUN_ORDER
                pos += 8
    return order


def pack_tiles(W: np.ndarray) -> np.ndarray:
    N, K = W.shape
    order = _full_tile_order(W.dtype.itemsize)
    out = np.empty(N * K, dtype=W.dtype)
    for g in range((N + ROWS_PER_GROUP - 1) // ROWS_PER_GROUP):
        r0 = ROWS_PER_GROUP * g
        rows_g = min(ROWS_PER_GROUP, N - r0)
        for kt in range((K + K_TILE - 1) // K_TILE):
            k0 = K_TILE * kt
            len_kt = min(K_TILE, K - k0)
            off = tile_offset(N, K, g, kt)
            block = W[r0:r0 + rows_g, k0:k0 + len_kt].reshape(-1)
            if rows_g == ROWS_PER_GROUP and len_kt == K_TILE:
                block = block[order]
            out[off:off + rows_g * len_kt] = block
    return out


def unpack_tiles(Pk: np.ndarray, N: int, K: int) -> np.ndarray:
    order = _full_tile_order(Pk.dtype.itemsize)
    W = np.empty((N, K), dtype=Pk.dtype)
    for g in range((N + ROWS_PER_GROUP - 1) // ROWS_PER_GROUP):
        r0 = ROWS_PER_GROUP * g
        rows_g = min(ROWS_PER_GROUP, N - r0)
        for kt in range((K + K_TILE - 1) // K_TILE):
            k0 = K_TILE * kt
            len_kt = min(K_TILE, K - k0)
            off = tile_offset(N, K, g, kt)
            block = Pk[off:off + rows_g * len_kt]
            if rows_g == ROWS_PER_GROUP and len_kt == K_TILE:
                flat = np.empty_like(block)
                flat[order] = block
                block = flat
            W[r0:r0 + rows_g, k0:k0 + len_kt] = block.reshape(rows_g, len_kt)
    return W
