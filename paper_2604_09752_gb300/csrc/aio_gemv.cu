// aio_gemv.cu -- instantiates the stream kernel for the plain step (every x an input) and the
// read probe, and holds the launch helpers (the kernel itself is in aio_stream.cuh).
#include "aio_stream.cuh"

namespace aio {
namespace {

// ------------------------------------------------------------------ read probe
// Same per-warp ring and slot size as the stream kernel, no arithmetic: each warp streams a
// contiguous range of 4 KB pages in slot-sized copies and folds word (lane * 32) of every page
// into *out.  Measures the read ceiling of the bulk-copy ring.
__global__ void __launch_bounds__(kThreads, 1) aio_probe_kernel(const uint8_t* buf, long long pages, unsigned* out) {
    constexpr int kPage = 4096, kPagesPerSlot = kSlotBytes / kPage;
    extern __shared__ __align__(1024) uint8_t smem[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    uint8_t* ring = smem + warp * kRingBytesPerWarp;
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kWarps * kRingBytesPerWarp) + warp * kMaxStages;
    const long long Z = static_cast<long long>(gridDim.x) * kWarps;
    const long long z = static_cast<long long>(blockIdx.x) * kWarps + warp;
    const long long p0 = seg_start(z, static_cast<int>(Z), pages);
    const long long p1 = seg_start(z + 1, static_cast<int>(Z), pages);
    if (lane == 0) {
        for (int i = 0; i < kStages; ++i) mbar_init(&bars[i], 1);
        fence_mbar_init();
    }
    __syncwarp();
    const uint64_t pol = policy_evict_first();
    long long ip = p0;        // next page to issue
    int islot = 0, in_flight = 0;
    auto issue = [&]() -> bool {
        if (ip >= p1) return false;
        const int n = static_cast<int>(min(static_cast<long long>(kPagesPerSlot), p1 - ip));
        if (lane == 0) {
            mbar_expect_tx(&bars[islot], static_cast<uint32_t>(n * kPage));
            bulk_g2s(ring + islot * kSlotBytes, buf + ip * kPage, static_cast<uint32_t>(n * kPage), &bars[islot], pol);
        }
        ip += n;
        islot = (islot + 1 == kStages) ? 0 : islot + 1;
        return true;
    };
    for (int i = 0; i < kStages; ++i)
        if (issue()) ++in_flight;
    unsigned acc = 0;
    int cslot = 0;
    uint32_t cphase = 0;
    for (long long pc = p0; pc < p1;) {
        if (!__all_sync(0xffffffffu, mbar_wait(&bars[cslot], cphase, 1000000000ull))) {
            for (int j = 0; j < in_flight; ++j) {   // bounded drain of this warp's copies, then leave
                mbar_wait(&bars[cslot], cphase, 1000000000ull);
                cslot = (cslot + 1 == kStages) ? 0 : cslot + 1;
                cphase ^= (cslot == 0) ? 1u : 0u;
            }
            return;
        }
        const int n = static_cast<int>(min(static_cast<long long>(kPagesPerSlot), p1 - pc));
        for (int j = 0; j < n; ++j)
            acc ^= reinterpret_cast<const unsigned*>(ring + cslot * kSlotBytes + j * kPage)[lane * 32];
        pc += n;
        __syncwarp();
        if (lane == 0) fence_proxy_async_smem();
        cslot = (cslot + 1 == kStages) ? 0 : cslot + 1;
        cphase ^= (cslot == 0) ? 1u : 0u;
        if (!issue()) --in_flight;
    }
    for (int o = 16; o; o >>= 1) acc ^= __shfl_xor_sync(0xffffffffu, acc, o);
    if (lane == 0) atomicXor(out, acc);
}

template <bool I8>
StreamFn stream_fn(int M) {
    switch (M) {
        case 1: return aio_stream_kernel<1, I8, false>;
        case 2: return aio_stream_kernel<2, I8, false>;
        case 3: return aio_stream_kernel<3, I8, false>;
        case 4: return aio_stream_kernel<4, I8, false>;
        case 5: return aio_stream_kernel<5, I8, false>;
        case 6: return aio_stream_kernel<6, I8, false>;
        case 7: return aio_stream_kernel<7, I8, false>;
        case 8: return aio_stream_kernel<8, I8, false>;
        default: return nullptr;
    }
}

StreamFn kernel_for(bool i8, int M, bool chained, bool phases) {
    if (chained) return chain_stream_fn(i8, M, phases);
    return i8 ? stream_fn<true>(M) : stream_fn<false>(M);
}

}  // namespace

cudaError_t prepare_kernels() {
    for (int ch = 0; ch < 3; ++ch) {   // plain, chained, chained with phases
        for (int i8 = 0; i8 < 2; ++i8) {
            for (int M = 1; M <= (ch ? kMaxChainM : kMaxM); ++M) {
                StreamFn f = kernel_for(i8 != 0, M, ch != 0, ch == 2);
                cudaError_t e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
                if (e != cudaSuccess) return e;
            }
        }
    }
    const cudaError_t e = cudaFuncSetAttribute(aio_probe_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
    return e != cudaSuccess ? e : prepare_small_kernels();
}

cudaError_t launch_stream(const StreamArgs& a, bool i8, int grid, cudaStream_t s, bool pdl, bool coop, bool chained,
                          bool phases) {
    StreamFn f = kernel_for(i8, a.M, chained, phases);
    if (!f) return cudaErrorInvalidValue;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(grid));
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = kSmemBytes;
    cfg.stream = s;
    cudaLaunchAttribute attr[2];
    int n = 0;
    if (pdl) {
        attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[n].val.programmaticStreamSerializationAllowed = 1;
        ++n;
    }
    if (coop) {
        attr[n].id = cudaLaunchAttributeCooperative;
        attr[n].val.cooperative = 1;
        ++n;
    }
    cfg.attrs = attr;
    cfg.numAttrs = n;
    return cudaLaunchKernelEx(&cfg, f, a);
}

cudaError_t occupancy(bool i8, int M, bool chained, bool phases, int* blocks_per_sm) {
    StreamFn f = kernel_for(i8, M, chained, phases);
    if (!f) return cudaErrorInvalidValue;
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(blocks_per_sm, f, kThreads, kSmemBytes);
}

cudaError_t launch_probe(const void* buf, long long pages, unsigned* out, int grid, cudaStream_t s) {
    aio_probe_kernel<<<grid, kThreads, kSmemBytes, s>>>(static_cast<const uint8_t*>(buf), pages, out);
    return cudaGetLastError();
}

}  // namespace aio
