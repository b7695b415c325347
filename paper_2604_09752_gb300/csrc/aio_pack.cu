// aio_pack.cu -- weight packer: row-major W [N, K] <-> tiled layout (8 rows x 256 k tiles).
//
// The packed layout makes every tile one contiguous block so the linear kernel streams it with
// a single bulk copy.  It is a pure permutation (no padding, bit-identical elements).  One
// thread moves one 16-byte piece (8 bf16 or 16 int8 elements), which never straddles a tile
// row because K % 16 == 0; reads of the row-major side are fully coalesced.
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
        const size_t packed = static_cast<size_t>(g) * kRows * K + static_cast<size_t>(kt) * rows * kKT +
                              static_cast<size_t>(r) * klen + kk;
        const size_t rowmajor = static_cast<size_t>(n) * K + k;
        if (INVERSE) {
            *reinterpret_cast<uint4*>(dst + rowmajor * E) = *reinterpret_cast<const uint4*>(src + packed * E);
        } else {
            *reinterpret_cast<uint4*>(dst + packed * E) = *reinterpret_cast<const uint4*>(src + rowmajor * E);
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
