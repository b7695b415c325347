// aio_gemv.cu -- the decode-step linear kernel: y = x W^T for M = 1..8 token rows,
// bf16 weights or int8 codes with per-output-channel bf16 scales (Sec. 2.1, Sec. 2.4).
//
// The work is a stream of weight bytes from HBM with 1 (bf16) or 2 (int8) FMAs per byte per
// token row, so the kernel is built around keeping enough bytes in flight:
//
//   * Weights are cut into tiles of 8 rows x 256 k (4 KB bf16, 2 KB int8), each one contiguous
//     block in the packed layout.  The T tiles of a matrix are split evenly over the Z warps of
//     the grid: warp z streams tiles [z*T/Z, (z+1)*T/Z), so every warp (and CTA) moves the same
//     number of bytes to within one tile, whatever N and K are.
//   * Each warp owns a 12 KB ring in shared memory.  Lane 0 issues one cp.async.bulk per tile
//     (global -> shared, L2 evict-first), completing on that slot's mbarrier; the warp waits on
//     the mbarrier (bounded by %globaltimer), computes, and refills the slot.  No producer warp,
//     no inter-warp synchronisation on the hot loop.
//   * Lane j owns k-columns [8j, 8j+8) of every tile; it keeps 8 rows x M accumulators in
//     registers and loads its 8 x values per row of x once per tile (reused by 8 weight rows).
//     bf16 -> fp32 is a shift/mask; int8 -> fp32 is exact via a byte permute into the mantissa
//     of 2^23 and one subtraction.  The int8 scale multiplies the finished fp32 sum.
//   * A row group whose tiles all lie in one warp's segment is reduced across lanes (shuffles)
//     and written directly.  A row group split between warps is finished by the last warp to
//     add its tile count to the group's counter: every contributor stores its partial sums,
//     fences, and bumps the counter; the last one sums all partials in warp order (so the
//     result is deterministic), writes y and resets the counter to zero.  Nothing spins.
//   * Programmatic dependent launch: the kernel signals its dependents at entry and issues its
//     first weight copies before griddepcontrol.wait, so it prefetches W while the previous
//     kernel on the stream finishes; x, y and the workspace are touched only after the wait.
#include <cuda_runtime.h>
#include <stdint.h>

#include "aio_internal.h"

namespace aio {
namespace {

// ------------------------------------------------------------------ PTX wrappers
__device__ __forceinline__ uint32_t smem_addr(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_mbar_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)), "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_addr(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// Bounded wait on a phase of an mbarrier; false if limit_ns elapsed first.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, unsigned long long limit_ns) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t start = globaltimer_ns();
    while (true) {
        if (mbar_try_wait(bar, parity)) return true;
        if (globaltimer_ns() - start > limit_ns) return false;
    }
}

__device__ __forceinline__ uint64_t policy_evict_first() {
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
    return p;
}

__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar, uint64_t pol) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;"
        ::"r"(smem_addr(dst)), "l"(src), "r"(bytes), "r"(smem_addr(bar)), "l"(pol)
        : "memory");
}

__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void griddep_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// ------------------------------------------------------------------ element helpers
__device__ __forceinline__ void bf16x8_to_f32(const uint4 v, float (&f)[8]) {
    f[0] = __uint_as_float(v.x << 16); f[1] = __uint_as_float(v.x & 0xFFFF0000u);
    f[2] = __uint_as_float(v.y << 16); f[3] = __uint_as_float(v.y & 0xFFFF0000u);
    f[4] = __uint_as_float(v.z << 16); f[5] = __uint_as_float(v.z & 0xFFFF0000u);
    f[6] = __uint_as_float(v.w << 16); f[7] = __uint_as_float(v.w & 0xFFFF0000u);
}

// int8 codes -> exact fp32.  (q ^ 0x80) is q + 128 as an unsigned byte u; placed in the low
// mantissa byte of 2^23 it reads as 2^23 + u, and subtracting 2^23 + 128 gives q exactly.
__device__ __forceinline__ void i8x8_to_f32(const uint2 v, float (&f)[8]) {
    const uint32_t a = v.x ^ 0x80808080u, b = v.y ^ 0x80808080u;
    const float bias = 8388736.0f;  // 2^23 + 128
    f[0] = __uint_as_float(__byte_perm(a, 0x4B000000u, 0x7440)) - bias;
    f[1] = __uint_as_float(__byte_perm(a, 0x4B000000u, 0x7441)) - bias;
    f[2] = __uint_as_float(__byte_perm(a, 0x4B000000u, 0x7442)) - bias;
    f[3] = __uint_as_float(__byte_perm(a, 0x4B000000u, 0x7443)) - bias;
    f[4] = __uint_as_float(__byte_perm(b, 0x4B000000u, 0x7440)) - bias;
    f[5] = __uint_as_float(__byte_perm(b, 0x4B000000u, 0x7441)) - bias;
    f[6] = __uint_as_float(__byte_perm(b, 0x4B000000u, 0x7442)) - bias;
    f[7] = __uint_as_float(__byte_perm(b, 0x4B000000u, 0x7443)) - bias;
}

__device__ __forceinline__ float bf16_to_f32(uint16_t h) { return __uint_as_float(static_cast<uint32_t>(h) << 16); }

template <bool I8>
struct TileT {
    static constexpr int kEsize = I8 ? 1 : 2;
    static constexpr int kBytes = kRows * kKT * kEsize;       // 2048 or 4096
    static constexpr int kStages = kRingBytesPerWarp / kBytes;  // 6 or 3
    static_assert(kStages <= kMaxStages, "ring slots exceed the barrier area");
};

struct TileCoord {
    int g, kt, rows, klen;
};

__device__ __forceinline__ TileCoord tile_coord(const GemvArgs& a, long long t) {
    TileCoord c;
    c.g = static_cast<int>(t / a.NKT);
    c.kt = static_cast<int>(t - static_cast<long long>(c.g) * a.NKT);
    c.rows = min(kRows, a.N - c.g * kRows);
    c.klen = min(kKT, a.K - c.kt * kKT);
    return c;
}

// Lane 0: arm the slot's barrier with the tile's byte count and issue its bulk copy (or, for
// row-major weights, one copy per row of the tile).
template <bool I8>
__device__ __forceinline__ void issue_tile(const GemvArgs& a, long long t, uint8_t* dst, uint64_t* bar,
                                           uint64_t pol) {
    constexpr int E = TileT<I8>::kEsize;
    const TileCoord c = tile_coord(a, t);
    const uint32_t bytes = static_cast<uint32_t>(c.rows * c.klen * E);
    mbar_expect_tx(bar, bytes);
    if (!a.rowmajor) {
        const size_t off = (static_cast<size_t>(c.g) * kRows * a.K + static_cast<size_t>(c.kt) * c.rows * kKT) * E;
        bulk_g2s(dst, a.w + off, bytes, bar, pol);
    } else {
        for (int r = 0; r < c.rows; ++r) {
            const size_t off = (static_cast<size_t>(c.g * kRows + r) * a.K + static_cast<size_t>(c.kt) * kKT) * E;
            bulk_g2s(dst + r * c.klen * E, a.w + off, static_cast<uint32_t>(c.klen * E), bar, pol);
        }
    }
}

// acc[r][m] += sum over this lane's 8 columns of W[row r] * x[m]
template <int MT, bool I8>
__device__ __forceinline__ void tile_fma(float (&acc)[kRows][MT], const uint8_t* tile, const TileCoord& c,
                                         int lane, const GemvArgs& a) {
    constexpr int E = TileT<I8>::kEsize;
    if (lane * 8 >= c.klen) return;
    float xf[MT][8];
    const uint16_t* xp = a.x + static_cast<size_t>(c.kt) * kKT + lane * 8;
#pragma unroll
    for (int m = 0; m < MT; ++m) {
        const uint4 v = *reinterpret_cast<const uint4*>(xp + static_cast<size_t>(m) * a.K);
        bf16x8_to_f32(v, xf[m]);
    }
    const uint8_t* base = tile + lane * 8 * E;
#pragma unroll
    for (int r = 0; r < kRows; ++r) {
        if (r < c.rows) {
            float wf[8];
            if constexpr (I8) {
                i8x8_to_f32(*reinterpret_cast<const uint2*>(base + r * c.klen), wf);
            } else {
                bf16x8_to_f32(*reinterpret_cast<const uint4*>(base + r * c.klen * 2), wf);
            }
#pragma unroll
            for (int m = 0; m < MT; ++m) {
#pragma unroll
                for (int e = 0; e < 8; ++e) acc[r][m] = fmaf(wf[e], xf[m][e], acc[r][m]);
            }
        }
    }
}

template <bool I8>
__device__ __forceinline__ float row_scale(const GemvArgs& a, int n) {
    if constexpr (I8) {
        return bf16_to_f32(a.scales[n]);
    } else {
        return 1.0f;
    }
}

// Warp z has finished its tiles of row group g (kt in [kt_lo, kt_hi]): reduce over lanes and
// either write y (group complete in this warp) or hand the partial to the last-arriver fixup.
template <int MT, bool I8>
__device__ __forceinline__ void finish_group(const GemvArgs& a, float (&acc)[kRows][MT], const TileCoord& c,
                                             long long z, long long t0, long long t1, int lane) {
#pragma unroll
    for (int r = 0; r < kRows; ++r) {
#pragma unroll
        for (int m = 0; m < MT; ++m) {
            float v = acc[r][m];
            v += __shfl_xor_sync(0xffffffffu, v, 16);
            v += __shfl_xor_sync(0xffffffffu, v, 8);
            v += __shfl_xor_sync(0xffffffffu, v, 4);
            v += __shfl_xor_sync(0xffffffffu, v, 2);
            v += __shfl_xor_sync(0xffffffffu, v, 1);
            acc[r][m] = v;
        }
    }
    const long long gfirst = static_cast<long long>(c.g) * a.NKT;
    const int kt_lo = t0 > gfirst ? static_cast<int>(t0 - gfirst) : 0;
    const int kt_hi = static_cast<int>(min(static_cast<long long>(a.NKT - 1), t1 - 1 - gfirst));
    const int row0 = c.g * kRows;

    if (kt_lo == 0 && kt_hi == a.NKT - 1) {
#pragma unroll
        for (int r = 0; r < kRows; ++r) {
#pragma unroll
            for (int m = 0; m < MT; ++m) {
                if (((r * MT + m) & 31) == lane && r < c.rows)
                    a.y[static_cast<size_t>(m) * a.N + row0 + r] = acc[r][m] * row_scale<I8>(a, row0 + r);
            }
        }
        return;
    }

    // Split group: publish this warp's partial, then count tiles; the warp completing the
    // count owns the final sum.
    constexpr int V = kRows * MT;
    const int side = (c.g == static_cast<int>(t0 / a.NKT)) ? 0 : 1;
    float* mine = a.partial + (static_cast<size_t>(z) * 2 + side) * V;
#pragma unroll
    for (int r = 0; r < kRows; ++r) {
#pragma unroll
        for (int m = 0; m < MT; ++m) {
            if (((r * MT + m) & 31) == lane) mine[r * MT + m] = acc[r][m];
        }
    }
    __threadfence();
    __syncwarp();
    const unsigned ntk = static_cast<unsigned>(kt_hi - kt_lo + 1);
    unsigned prev = 0;
    if (lane == 0) prev = atomicAdd(&a.counters[c.g], ntk);
    prev = __shfl_sync(0xffffffffu, prev, 0);
    if (prev + ntk != static_cast<unsigned>(a.NKT)) return;

    __threadfence();
    const long long tf = gfirst, tl = gfirst + a.NKT - 1;
    const long long zf = ((tf + 1) * a.Z - 1) / a.T;   // warp whose segment holds tile tf
    const long long zl = ((tl + 1) * a.Z - 1) / a.T;   // ... and tile tl
    for (int v = lane; v < V; v += 32) {
        const int r = v / MT, m = v - (v / MT) * MT;
        if (r >= c.rows) continue;
        float sum = 0.0f;
        for (long long zz = zf; zz <= zl; ++zz) {
            const long long s0 = zz * a.T / a.Z, s1 = (zz + 1) * a.T / a.Z;
            if (s1 == s0) continue;
            const int sd = (c.g == static_cast<int>(s0 / a.NKT)) ? 0 : 1;
            sum += __ldcg(a.partial + (static_cast<size_t>(zz) * 2 + sd) * V + v);
        }
        a.y[static_cast<size_t>(m) * a.N + row0 + r] = sum * row_scale<I8>(a, row0 + r);
    }
    if (lane == 0) a.counters[c.g] = 0u;
}

template <int MT, bool I8>
__global__ void __launch_bounds__(kThreads, (MT <= 4) ? 2 : 1) aio_gemv_kernel(const GemvArgs a) {
    using TL = TileT<I8>;
    extern __shared__ __align__(1024) uint8_t smem[];
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    uint8_t* ring = smem + warp * kRingBytesPerWarp;
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kWarps * kRingBytesPerWarp) + warp * kMaxStages;

    griddep_launch_dependents();

    const long long z = static_cast<long long>(blockIdx.x) * kWarps + warp;
    const long long t0 = z * a.T / a.Z;
    const long long t1 = (z + 1) * a.T / a.Z;
    const int ntiles = static_cast<int>(t1 - t0);

    if (lane == 0) {
#pragma unroll
        for (int s = 0; s < TL::kStages; ++s) mbar_init(&bars[s], 1);
        fence_mbar_init();
    }
    __syncwarp();

    const uint64_t pol = policy_evict_first();
    const bool stall = a.test_stall && z == a.Z - 1;  // the grid's last warp always owns >= 1 tile
    if (lane == 0) {
        const int npro = min(ntiles, TL::kStages);
        for (int i = 0; i < npro; ++i) {
            if (stall && i == 0) continue;  // test hook: this slot's barrier never completes
            issue_tile<I8>(a, t0 + i, ring + i * TL::kBytes, &bars[i], pol);
        }
    }

    // Everything below reads x / writes y and the workspace: wait for the previous grid.
    griddep_wait();

    float acc[kRows][MT];
#pragma unroll
    for (int r = 0; r < kRows; ++r)
#pragma unroll
        for (int m = 0; m < MT; ++m) acc[r][m] = 0.0f;

    for (int i = 0; i < ntiles; ++i) {
        const long long t = t0 + i;
        const int s = i % TL::kStages;
        const uint32_t parity = static_cast<uint32_t>(i / TL::kStages) & 1u;
        const bool ok = __all_sync(0xffffffffu, mbar_wait(&bars[s], parity, a.wait_limit_ns));
        if (!ok) {
            // Record the timeout, then wait (bounded) for this warp's other copies in flight so
            // no bulk copy targets shared memory after the CTA exits.
            if (lane == 0) atomicExch(a.err, kDevErrTimeout);
            const int last_issued = min(ntiles, i + TL::kStages);
            for (int j = i; j < last_issued; ++j)
                mbar_wait(&bars[j % TL::kStages], static_cast<uint32_t>(j / TL::kStages) & 1u, a.wait_limit_ns);
            return;
        }
        const TileCoord c = tile_coord(a, t);
        tile_fma<MT, I8>(acc, ring + s * TL::kBytes, c, lane, a);
        __syncwarp();
        if (lane == 0 && i + TL::kStages < ntiles) {
            fence_proxy_async_smem();  // order this warp's reads of the slot before the refill
            issue_tile<I8>(a, t + TL::kStages, ring + s * TL::kBytes, &bars[s], pol);
        }
        if (c.kt == a.NKT - 1 || i == ntiles - 1) {
            finish_group<MT, I8>(a, acc, c, z, t0, t1, lane);
#pragma unroll
            for (int r = 0; r < kRows; ++r)
#pragma unroll
                for (int m = 0; m < MT; ++m) acc[r][m] = 0.0f;
        }
    }
}

// ------------------------------------------------------------------ read probe
// Same per-warp ring as the linear kernel, 4 KB chunks, one word per chunk folded into *out.
__global__ void __launch_bounds__(kThreads, 2) aio_probe_kernel(const uint8_t* buf, long long chunks, unsigned* out) {
    constexpr int kChunk = 4096, kStages = kRingBytesPerWarp / kChunk;
    extern __shared__ __align__(1024) uint8_t smem[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    uint8_t* ring = smem + warp * kRingBytesPerWarp;
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kWarps * kRingBytesPerWarp) + warp * kMaxStages;
    const long long Z = static_cast<long long>(gridDim.x) * kWarps;
    const long long z = static_cast<long long>(blockIdx.x) * kWarps + warp;
    const long long c0 = z * chunks / Z, c1 = (z + 1) * chunks / Z;
    const int n = static_cast<int>(c1 - c0);
    if (lane == 0) {
        for (int s = 0; s < kStages; ++s) mbar_init(&bars[s], 1);
        fence_mbar_init();
    }
    __syncwarp();
    const uint64_t pol = policy_evict_first();
    if (lane == 0) {
        for (int i = 0; i < min(n, kStages); ++i) {
            mbar_expect_tx(&bars[i], kChunk);
            bulk_g2s(ring + i * kChunk, buf + (c0 + i) * kChunk, kChunk, &bars[i], pol);
        }
    }
    unsigned acc = 0;
    for (int i = 0; i < n; ++i) {
        const int s = i % kStages;
        if (!__all_sync(0xffffffffu, mbar_wait(&bars[s], static_cast<uint32_t>(i / kStages) & 1u, 1000000000ull))) {
            for (int j = i + 1; j < min(n, i + kStages); ++j)
                mbar_wait(&bars[j % kStages], static_cast<uint32_t>(j / kStages) & 1u, 1000000000ull);
            return;
        }
        acc ^= reinterpret_cast<const unsigned*>(ring + s * kChunk)[lane * 32];
        __syncwarp();
        if (lane == 0 && i + kStages < n) {
            fence_proxy_async_smem();
            mbar_expect_tx(&bars[s], kChunk);
            bulk_g2s(ring + s * kChunk, buf + (c0 + i + kStages) * kChunk, kChunk, &bars[s], pol);
        }
    }
    for (int o = 16; o; o >>= 1) acc ^= __shfl_xor_sync(0xffffffffu, acc, o);
    if (lane == 0) atomicXor(out, acc);
}

using GemvFn = void (*)(const GemvArgs);

template <bool I8>
GemvFn gemv_fn(int M) {
    switch (M) {
        case 1: return aio_gemv_kernel<1, I8>;
        case 2: return aio_gemv_kernel<2, I8>;
        case 3: return aio_gemv_kernel<3, I8>;
        case 4: return aio_gemv_kernel<4, I8>;
        case 5: return aio_gemv_kernel<5, I8>;
        case 6: return aio_gemv_kernel<6, I8>;
        case 7: return aio_gemv_kernel<7, I8>;
        case 8: return aio_gemv_kernel<8, I8>;
        default: return nullptr;
    }
}

}  // namespace

cudaError_t prepare_kernels() {
    for (int i8 = 0; i8 < 2; ++i8) {
        for (int M = 1; M <= kMaxM; ++M) {
            GemvFn f = i8 ? gemv_fn<true>(M) : gemv_fn<false>(M);
            cudaError_t e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
            if (e != cudaSuccess) return e;
        }
    }
    return cudaFuncSetAttribute(aio_probe_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
}

cudaError_t launch_gemv(const GemvArgs& a, bool i8, int grid, cudaStream_t s, bool pdl) {
    GemvFn f = i8 ? gemv_fn<true>(a.M) : gemv_fn<false>(a.M);
    if (!f) return cudaErrorInvalidValue;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(grid));
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = kSmemBytes;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, f, a);
}

cudaError_t launch_probe(const void* buf, long long chunks, unsigned* out, int grid, cudaStream_t s) {
    aio_probe_kernel<<<grid, kThreads, kSmemBytes, s>>>(static_cast<const uint8_t*>(buf), chunks, out);
    return cudaGetLastError();
}

}  // namespace aio
