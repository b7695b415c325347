// aio_pack.cu -- weight packer: row-major W [N, K] <-> tiled layout.
//
// Tiles are 8 rows x 256 k; consecutive tiles are contiguous, so any run of them is one bulk copy.
// A full tile (8 rows, 256 k) is stored in the order the stream kernel's lanes read it: 16-byte
// piece j of lane L = 4 r + c holds W[row r][64 c + j * (8 bf16 | 16 int8) ...], at byte
// j * 512 + L * 16 of the tile, so every 128-bit shared-memory load of a warp is contiguous.
// Ragged tiles (last row group or last k tile) stay row-major.  The layout is a pure permutation
// (no padding); one thread moves one 16-byte piece, and the row-major side is fully coalesced.
#include <cuda_runtime.h>
#include <stdint.h>

#include "aio_internal.h"

namespace aio {
namespace {

template <int E, bool INVERSE>
__global__ void __launch_bounds__(256) aio_pack_kernel(const uint8_t* __restrict__ src, uint8_t* __restrict__ dst,
                                                       int N, int K) {
    constexpr int kPiece = 16 / E;                 // elements per 16-byte piece
    const long long per_row = K / kPiece;
    const long long total = static_cast<long long>(N) * per_row;
    for (long long p = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x; p < total;
         p += static_cast<long long>(gridDim.x) * blockDim.x) {
        const int n = static_cast<int>(p / per_row);
        const int k = static_cast<int>(p - static_cast<long long>(n) * per_row) * kPiece;
        const int g = n / kRows, r = n - g * kRows;
        const int kt = k / kKT, kk = k - kt * kKT;
        const int rows = min(kRows, N - g * kRows);
        const int klen = min(kKT, K - kt * kKT);
        const size_t tile = (static_cast<size_t>(g) * kRows * K + static_cast<size_t>(kt) * rows * kKT) * E;
        size_t in_tile;
        if (rows == kRows && klen == kKT) {
            const int c = kk / 64, j = (kk - 64 * c) / kPiece;
            in_tile = static_cast<size_t>(j) * 512 + (r * 4 + c) * 16;
        } else {
            in_tile = (static_cast<size_t>(r) * klen + kk) * E;
        }
        const size_t packed = tile + in_tile;
        const size_t rowmajor = (static_cast<size_t>(n) * K + k) * E;
        if (INVERSE) {
            *reinterpret_cast<uint4*>(dst + rowmajor) = *reinterpret_cast<const uint4*>(src + packed);
        } else {
            *reinterpret_cast<uint4*>(dst + packed) = *reinterpret_cast<const uint4*>(src + rowmajor);
        }
    }
}

}  // namespace

cudaError_t launch_pack(const void* src, void* dst, int N, int K, int esize, bool inverse, cudaStream_t s) {
    const long long pieces = static_cast<long long>(N) * K * esize / 16;
    const int block = 256;
    long long grid = (pieces + block - 1) / block;
    if (grid > 65535LL * 16) grid = 65535LL * 16;
    if (grid < 1) grid = 1;
    const uint8_t* a = static_cast<const uint8_t*>(src);
    uint8_t* b = static_cast<uint8_t*>(dst);
    const unsigned g = static_cast<unsigned>(grid);
    if (esize == 2) {
        if (inverse) aio_pack_kernel<2, true><<<g, block, 0, s>>>(a, b, N, K);
        else aio_pack_kernel<2, false><<<g, block, 0, s>>>(a, b, N, K);
    } else {
        if (inverse) aio_pack_kernel<1, true><<<g, block, 0, s>>>(a, b, N, K);
        else aio_pack_kernel<1, false><<<g, block, 0, s>>>(a, b, N, K);
    }
    return cudaGetLastError();
}

}  // namespace aio
