"""Reference definition of the tiled weight layout (TEST INFRASTRUCTURE).

The CUDA packer reorders W [N, K] (bf16 or int8) so that each streamed tile
is one contiguous block of bytes.  The layout is a pure permutation of the
elements, written here with plain numpy loops so the GPU packer can be checked
bit for bit against it:

  * rows are grouped 8 at a time: row group g holds rows [8g, 8g + rows_g),
    rows_g = min(8, N - 8g); the group starts at element offset 8 g K;
  * inside a group, k is cut into tiles of 256 columns: tile kt covers
    [256 kt, 256 kt + len_kt), len_kt = min(256, K - 256 kt), and starts at
    element offset rows_g * 256 * kt from the start of its group;
  * inside a tile the block is row-major [rows_g, len_kt].

No padding is added, so the packed buffer has exactly N*K elements.
"""
from __future__ import annotations

import numpy as np

ROWS_PER_GROUP = 8
K_TILE = 256


def tile_offset(N: int, K: int, g: int, kt: int) -> int:
    rows_g = min(ROWS_PER_GROUP, N - ROWS_PER_GROUP * g)
    return ROWS_PER_GROUP * g * K + rows_g * K_TILE * kt


def pack_tiles(W: np.ndarray) -> np.ndarray:
    N, K = W.shape
    out = np.empty(N * K, dtype=W.dtype)
    for g in range((N + ROWS_PER_GROUP - 1) // ROWS_PER_GROUP):
        r0 = ROWS_PER_GROUP * g
        rows_g = min(ROWS_PER_GROUP, N - r0)
        for kt in range((K + K_TILE - 1) // K_TILE):
            k0 = K_TILE * kt
            len_kt = min(K_TILE, K - k0)
            off = tile_offset(N, K, g, kt)
            out[off:off + rows_g * len_kt] = W[r0:r0 + rows_g, k0:k0 + len_kt].reshape(-1)
    return out


def unpack_tiles(P: np.ndarray, N: int, K: int) -> np.ndarray:
    W = np.empty((N, K), dtype=P.dtype)
    for g in range((N + ROWS_PER_GROUP - 1) // ROWS_PER_GROUP):
        r0 = ROWS_PER_GROUP * g
        rows_g = min(ROWS_PER_GROUP, N - r0)
        for kt in range((K + K_TILE - 1) // K_TILE):
            k0 = K_TILE * kt
            len_kt = min(K_TILE, K - k0)
            off = tile_offset(N, K, g, kt)
            W[r0:r0 + rows_g, k0:k0 + len_kt] = P[off:off + rows_g * len_kt].reshape(rows_g, len_kt)
    return W
