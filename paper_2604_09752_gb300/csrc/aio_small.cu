// aio_small.cu -- a small projection launched on its own: y = x W^T (Sec. 2.1; int8 codes with
// per-channel scales, Sec. 2.4) when the whole matrix is a few MB, as the single 2048 x 2048 layer
// of a 1B-class decoder is (8 MB).
//
// Launched alone, such a projection is bound by latency, not by HBM bandwidth: the stream kernel
// spreads its ~1000 tiles over 1216 warps, so every row group is split across several warps and its
// partial sums meet in global memory, one more round trip after the weights land; and its 227 KB
// CTAs keep the next launch off the SMs until they exit.  Here one CTA takes one row group:
//   * warp w streams tiles [w NKT / 8, (w + 1) NKT / 8) of the group with one bulk copy, issued
//     before griddepcontrol.wait, so the weights load while the previous kernel on the stream ends;
//   * the eight warps' partial sums meet in shared memory and are added in warp order (the result
//     does not depend on timing); then 16 M threads scale and store y;
//   * a CTA needs at most 96 KB of shared memory, so two fit an SM and a launch chained with
//     programmatic dependent launch starts its copies beside the previous one.
// x is read from global memory (L2: every CTA reads the same M rows).
#include "aio_stream.cuh"

namespace aio {
namespace {

constexpr int kSmallRedBytes = kWarps * kRows * kMaxM * 4;   // the warps' partial sums
constexpr int kSmallMaxTileBytes = 96 * 1024;                // weights of one CTA

template <int MT, bool I8>
__global__ void __launch_bounds__(kThreads, 2) aio_small_kernel(const __grid_constant__ StreamArgs s, int tpw) {
    using TL = TileT<I8>;
    constexpr int E = TL::kEsize;
    griddep_launch_dependents();
    extern __shared__ __align__(1024) uint8_t smem[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const ProjDesc& D = s.one;
    const int K = D.K, N = D.N, NKT = D.NKT;
    const int g = blockIdx.x;                                  // this CTA's row group
    const int rows = min(kRows, N - g * kRows);
    const int kt0 = warp * NKT / kWarps, kt1 = (warp + 1) * NKT / kWarps;   // this warp's tiles of it
    uint8_t* wbuf = smem + static_cast<size_t>(warp) * tpw * TL::kBytes;
    uint64_t* bar = reinterpret_cast<uint64_t*>(smem + static_cast<size_t>(kWarps) * tpw * TL::kBytes) + warp;
    float* red = reinterpret_cast<float*>(smem + static_cast<size_t>(kWarps) * tpw * TL::kBytes + kWarps * 8);
    if (lane == 0) {
        mbar_init(bar, 1);
        fence_mbar_init();
    }
    __syncwarp();
    // the test hook: the grid's last warp skips its copy, so its bounded wait expires
    const bool stall = s.test_stall && g == static_cast<int>(gridDim.x) - 1 && warp == kWarps - 1;
    const bool any = kt1 > kt0;
    if (any && lane == 0 && !stall) {
        const size_t off = tile_offset<E>(K, N, g, kt0);
        const size_t end = tile_offset<E>(K, N, g, kt1 - 1) + static_cast<size_t>(rows) * min(kKT, K - (kt1 - 1) * kKT) * E;
        mbar_expect_tx(bar, static_cast<uint32_t>(end - off));
        bulk_g2s(wbuf, D.w + off, static_cast<uint32_t>(end - off), bar, policy_evict_first());
    }
    // x, y and the error word wait for the previous kernel on the stream
    griddep_wait();

    const Proj P = load_proj<false>(&D, MT);
    [[maybe_unused]] const I8Consts kc = i8_consts();
    float d[4][4] = {};
    bool ok = true;
    if (any) {
        ok = __all_sync(0xffffffffu, mbar_wait(bar, 0, s.wait_limit_ns));
        if (ok) {
            const int tok = lane >> 2, xtok = min(tok, MT - 1);
            const uint16_t* xrow = P.x + static_cast<size_t>(tok) * K;                             // ragged tiles
            [[maybe_unused]] const uint16_t* xlane = P.x + static_cast<size_t>(xtok) * K + 8 * (lane & 3);   // full tiles
            const uint8_t* tp = wbuf;
            for (int kt = kt0; kt < kt1; ++kt) {
                const int klen = min(kKT, K - kt * kKT);
                if (rows == kRows && klen == kKT) {
#if AIO_FFMA
                    ffma_full_g<I8, MT>(d, tp + lane * 16, P.x + 8 * (lane & 3) + kt * kKT, K);
#else
                    tile_mma_full<I8>(d, tp + lane * 16, xlane + kt * kKT, kc);
#endif
                } else {
                    tile_mma<I8>(d, tp, rows, klen, kt * kKT, lane, P, xrow, kc);
                }
                tp += static_cast<size_t>(rows) * klen * E;
            }
        } else if (lane == 0) {
            atomicExch(s.err, kDevErrTimeout);
            if (!stall) mbar_wait(bar, 0, s.wait_limit_ns);   // bounded: the copy in flight lands before exit
        }
    }
    // lane (r, c) holds D[row r + 8 (i / 2)][token 2c + i % 2] in sum[i]
    float sum[4];
#if AIO_FFMA
    ffma_finish<MT>(d, sum, lane);
#else
#pragma unroll
    for (int i = 0; i < 4; ++i) sum[i] = (d[0][i] + d[1][i]) + (d[2][i] + d[3][i]);
#endif
    const int gr = lane >> 2, m0 = 2 * (lane & 3);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int m = m0 + (i & 1), r = gr + 8 * (i >> 1);
        if (m < MT) red[(warp * MT + m) * kRows + r] = sum[i];
    }
    __syncthreads();
    const int t = threadIdx.x;
    if (t < kRows * MT) {
        const int m = t / kRows, r = t - m * kRows;
        if (r < rows) {
            float v = 0.0f;
#pragma unroll
            for (int w = 0; w < kWarps; ++w) v += red[(w * MT + m) * kRows + r];
            P.y[static_cast<size_t>(m) * N + g * kRows + r] = v * row_scale<I8>(P, g * kRows + r);
        }
    }
}

using SmallFn = void (*)(const StreamArgs, int);

template <bool I8>
SmallFn small_fn(int M) {
    switch (M) {
        case 1: return aio_small_kernel<1, I8>;
        case 2: return aio_small_kernel<2, I8>;
        case 3: return aio_small_kernel<3, I8>;
        case 4: return aio_small_kernel<4, I8>;
        case 5: return aio_small_kernel<5, I8>;
        case 6: return aio_small_kernel<6, I8>;
        case 7: return aio_small_kernel<7, I8>;
        case 8: return aio_small_kernel<8, I8>;
        default: return nullptr;
    }
}

}  // namespace

SmallGeometry small_geometry(int K, int N, bool i8, bool rowmajor, int num_sms) {
    SmallGeometry g = {};
    const int NG = (N + kRows - 1) / kRows, NKT = (K + kKT - 1) / kKT;
    g.tpw = (NKT + kWarps - 1) / kWarps;
    const int tile = i8 ? TileT<true>::kBytes : TileT<false>::kBytes;
    g.grid = NG;
    g.smem = static_cast<size_t>(kWarps) * g.tpw * tile + kWarps * 8 + kSmallRedBytes;
    g.ok = !rowmajor && NG <= 2 * num_sms && kWarps * g.tpw * tile <= kSmallMaxTileBytes;
    return g;
}

cudaError_t prepare_small_kernels() {
    for (int M = 1; M <= kMaxM; ++M) {
        for (SmallFn f : {small_fn<false>(M), small_fn<true>(M)}) {
            const cudaError_t e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                       kSmallMaxTileBytes + kWarps * 8 + kSmallRedBytes);
            if (e != cudaSuccess) return e;
        }
    }
    return cudaSuccess;
}

cudaError_t launch_small(const StreamArgs& a, bool i8, const SmallGeometry& g, cudaStream_t s, bool pdl) {
    SmallFn f = i8 ? small_fn<true>(a.M) : small_fn<false>(a.M);
    if (!f || !g.ok) return cudaErrorInvalidValue;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(g.grid));
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = g.smem;
    cfg.stream = s;
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr.val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = &attr;
    cfg.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, f, a, g.tpw);
}

}  // namespace aio
