"""Reference definition of the tiled weight layout (TEST INFRASTRUCTURE).

The CUDA packer reorders W [N, K] (bf16 or int8) into tiles so that each streamed run of tiles
is one contiguous block of bytes, and so that a full tile sits in shared memory in the order the
kernel's lanes read it.  The layout is a pure permutation of the elements, written here with
plain numpy slicing so the GPU packer can be checked bit for bit against it:

  * rows are grouped 8 at a time: row group g holds rows [8g, 8g + rows_g),
    rows_g = min(8, N - 8g); the group starts at element offset 8 g K;
  * inside a group, k is cut into tiles of 256 columns: tile kt covers
    [256 kt, 256 kt + len_kt), len_kt = min(256, K - 256 kt), and starts at
    element offset rows_g * 256 * kt from the start of its group;
  * a full tile (rows_g = 8, len_kt = 256) is stored as 16-byte pieces: piece j of lane
    L = 4 r + c (r = row in the tile, c = 0..3) holds the P consecutive elements
    W[r, 64 c + P j : 64 c + P (j + 1)] (P = 8 for 2-byte, 16 for 1-byte elements) and sits at
    byte j * 512 + L * 16 of the tile;
  * a ragged tile is the row-major block [rows_g, len_kt].

No padding is added, so the packed buffer has exactly N*K elements.
"""
from __future__ import annotations

import numpy as np

ROWS_PER_GROUP = 8
K_TILE = 256


def tile_offset(N: int, K: int, g: int, kt: int) -> int:
    rows_g = min(ROWS_PER_GROUP, N - ROWS_PER_GROUP * g)
    return ROWS_PER_GROUP * g * K + rows_g * K_TILE * kt


def _full_tile_order(esize: int) -> np.ndarray:
    """order[i] = row-major index (r * 256 + k) of the element stored at position i of a full tile."""
    P = 16 // esize                      # elements per 16-byte piece
    pieces = 256 // (4 * P)              # pieces per lane
    order = np.empty(ROWS_PER_GROUP * K_TILE, dtype=np.int64)
    for j in range(pieces):
        for L in range(32):
            r, c = divmod(L, 4)
            pos = (j * 512 + L * 16) // esize
            k0 = 64 * c + P * j
            order[pos:pos + P] = r * K_TILE + k0 + np.arange(P)
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
