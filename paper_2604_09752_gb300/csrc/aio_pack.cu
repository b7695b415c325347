// aio_pack.cu -- weight packer: row-major W [N, K] <-> tiled layout.
//
// Tiles are 16 rows x 256 k; consecutive tiles are contiguous, so any run of them is one bulk copy.
// A full tile (16 rows, 256 k) is stored in the order the stream kernel's lanes read it: lane
// L = 4 r + c (r = 0..7, c = 0..3) reads 16-byte piece j at byte j * 512 + 16 L of the tile:
//   bf16: piece s (0..15) is one MMA's A fragment for k-step s, k0 = 32 (s/2) + 8 c + 4 (s%2):
//         words W[r][k0..k0+1], W[r+8][k0..k0+1], W[r][k0+2..k0+3], W[r+8][k0+2..k0+3];
//   int8: pieces hold runs of 8 consecutive k, W[row][32 t + 8 c .. +8); piece j = 4 h + u holds
//         row r + 8 h, runs t = 2u (bytes 0-7) and t = 2u + 1 (bytes 8-15),
//         each 4-code word of a run stored as codes (0, 2, 1, 3): the first k pair in the low bytes
//         of the word's 16-bit halves, the second in the high bytes (the swap is its own inverse).
// Every 128-bit shared-memory load of a warp is then contiguous.  Ragged tiles (last row group or
// last k tile) stay row-major.  The layout is a pure permutation (no padding); one thread moves one
// 8-byte unit, and the row-major side is fully coalesced.
#include <cuda_runtime.h>
#include <stdint.h>

#include "aio_internal.h"

namespace aio {
namespace {

template <int E, bool INVERSE>
__global__ void __launch_bounds__(256) aio_pack_kernel(const uint8_t* __restrict__ src, uint8_t* __restrict__ dst,
                                                       int N, int K) {
    constexpr int kUnit = 8 / E;                   // elements per 8-byte unit
    const long long per_row = K / kUnit;
    const long long total = static_cast<long long>(N) * per_row;
    for (long long p = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x; p < total;
         p += static_cast<long long>(gridDim.x) * blockDim.x) {
        const int n = static_cast<int>(p / per_row);
        const int k = static_cast<int>(p - static_cast<long long>(n) * per_row) * kUnit;
        const int g = n / kRows, r = n - g * kRows;
        const int kt = k / kKT, kk = k - kt * kKT;
        const int rows = min(kRows, N - g * kRows);
        const int klen = min(kKT, K - kt * kKT);
        const size_t tile = (static_cast<size_t>(g) * kRows * K + static_cast<size_t>(kt) * rows * kKT) * E;
        const bool full = rows == kRows && klen == kKT;
        const size_t rowmajor = (static_cast<size_t>(n) * K + k) * E;
        if (E == 2 && full) {
            // 4 bf16 at k0 = kk: pair (k0, k0+1) is word h of piece s, pair (k0+2, k0+3) word 2 + h
            const int h = r >> 3, lane = (r & 7) * 4 + ((kk >> 3) & 3), s = 2 * (kk >> 5) + ((kk >> 2) & 1);
            uint8_t* piece = (INVERSE ? const_cast<uint8_t*>(src) : dst) + tile + static_cast<size_t>(s) * 512 + lane * 16;
            uint32_t* w0 = reinterpret_cast<uint32_t*>(piece) + h;
            uint32_t* w1 = reinterpret_cast<uint32_t*>(piece) + 2 + h;
            if (INVERSE) {
                *reinterpret_cast<uint2*>(dst + rowmajor) = make_uint2(*w0, *w1);
            } else {
                const uint2 v = *reinterpret_cast<const uint2*>(src + rowmajor);
                *w0 = v.x;
                *w1 = v.y;
            }
            continue;
        }
        size_t in_tile;
        if (full) {
            const int h = r >> 3, lane = (r & 7) * 4 + ((kk & 31) >> 3), t = kk >> 5;
            in_tile = static_cast<size_t>((kKT / 64) * h + (t >> 1)) * 512 + lane * 16 + (t & 1) * 8;
        } else {
            in_tile = (static_cast<size_t>(r) * klen + kk) * E;
        }
        const size_t packed = tile + in_tile;
        uint2 v = *reinterpret_cast<const uint2*>(src + (INVERSE ? packed : rowmajor));
        if (E == 1 && full) {   // swap bytes 1 and 2 of each word
            v.x = __byte_perm(v.x, 0u, 0x3120u);
            v.y = __byte_perm(v.y, 0u, 0x3120u);
        }
        *reinterpret_cast<uint2*>(dst + (INVERSE ? rowmajor : packed)) = v;
    }
}

}  // namespace

cudaError_t launch_pack(const void* src, void* dst, int N, int K, int esize, bool inverse, cudaStream_t s) {
    const long long units = static_cast<long long>(N) * K * esize / 8;
    const int block = 256;
    long long grid = (units + block - 1) / block;
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
