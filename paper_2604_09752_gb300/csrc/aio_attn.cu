// aio_attn.cu -- decode attention over a KV cache: the long-context half of the paper's routing
// (contexts up to 2K tokens are standard, up to 32K long: Sec. 3.3, Sec. 5.1).  For M new tokens
// at positions L - M .. L - 1 of a cache of L positions, per head h of dimension 128:
//   s_j = q[m, h] . k[h, j] / sqrt(128)   for j <= L - M + m,   out[m, h] = sum_j softmax(s)_j v[h, j].
//
// Like the projections, this streams bytes from HBM (2 * 256 B per position and head) with a few
// flops per byte, so it reuses the stream kernel's machinery: one CTA of 8 warps per SM, a ring of
// bulk copies per warp, and an even split of the work over all warps.
//   * Cache layout: [head][position][128] bf16, so a run of positions of one head is contiguous.
//   * Units: 16 positions of one head (4 KB of K and 4 KB of V, one ring slot).  The n_heads *
//     ceil(L / 16) units, head-major, are split evenly over the Z warps.  A warp's units span at
//     most two heads (n_heads <= Z), so it produces at most two partial results.
//   * Per unit: lane l holds dims [4l, 4l + 4) of q (fp32, scaled by log2(e) / sqrt(128)) for every
//     token.  The 16 partial dot products of a lane are reduced across the warp with 16 shuffles
//     (a transposing reduction: each halving step trades the half of the values a lane does not
//     keep), then the lane pair 2p, 2p + 1 holds position p's score.  An online softmax in base 2
//     keeps a running max, sum and weighted sum of V (lane l: dims [4l, 4l + 4)).
//   * A second small kernel merges each head's partials (max, sum, weighted V) in a fixed order, so
//     the result does not depend on timing.
//   * Both launch with programmatic dependent launch.  The partial kernel issues its first K and V
//     copies (the cache does not depend on earlier work on the stream) before it waits for the
//     previous kernel, then reads q and writes its partials; the merge kernel's small CTAs start
//     beside it and wait for it.  So one call's merge overlaps the next call's first copies.
#include "aio_attn.h"
#include "aio_stream.cuh"

namespace aio {
namespace {

// kHeadDim, kAttnPos (positions per unit), kAttnUnitBytes, kAttnSlot and kAttnRec (floats per
// partial: 128 weighted V, max, sum, pad) are shared with the chained step (aio_internal.h).
constexpr int kAttnStages = kRingBytesPerWarp / kAttnSlot;    // 3 slots of 8 KB per warp
constexpr int kAttnSmem = kWarps * kAttnStages * kAttnSlot + kWarps * kAttnStages * 8;
static_assert(kAttnStages >= 2, "attention ring");

struct AttnArgs {
    const float* q;           // [M, q_stride]
    const uint16_t* k;        // [n_heads][L_max][128]
    const uint16_t* v;
    float* out;               // [M, n_heads * 128]
    float* part;              // [Z][2][M][kAttnRec]
    int* err;
    int q_stride, n_heads, L_max, L, M, Z, nch;
    long long U;              // units = n_heads * nch
    unsigned long long wait_limit_ns;
};

__device__ __forceinline__ long long attn_seg(long long z, long long U, int Z) { return z * U / Z; }

template <int MT>
__global__ void __launch_bounds__(kThreads, 1) aio_attn_partial_kernel(const __grid_constant__ AttnArgs a) {
    griddep_launch_dependents();
    extern __shared__ __align__(1024) uint8_t smem[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    uint8_t* ring = smem + warp * kAttnStages * kAttnSlot;
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kWarps * kAttnStages * kAttnSlot) + warp * kAttnStages;
    const long long z = static_cast<long long>(blockIdx.x) * kWarps + warp;
    if (lane == 0) {
#pragma unroll
        for (int i = 0; i < kAttnStages; ++i) mbar_init(&bars[i], 1);
        fence_mbar_init();
    }
    __syncwarp();
    const long long u0 = attn_seg(z, a.U, a.Z), u1 = attn_seg(z + 1, a.U, a.Z);
    const uint64_t pol = policy_evict_first();

    // issue side: unit u -> head u / nch, positions [16 (u % nch), +16) clipped to L; the head and
    // chunk are tracked incrementally (one division per warp)
    long long ui = u0;
    int ih = static_cast<int>(u0 / a.nch), ic = static_cast<int>(u0 - static_cast<long long>(ih) * a.nch);
    auto issue = [&](int slot) {
        if (ui >= u1) return;
        const int h = ih, c = ic;
        if (++ic == a.nch) {
            ic = 0;
            ++ih;
        }
        const int p0 = c * kAttnPos, np = min(kAttnPos, a.L - p0);
        const uint32_t bytes = static_cast<uint32_t>(np * kHeadDim * 2);
        const size_t off = (static_cast<size_t>(h) * a.L_max + p0) * kHeadDim;
        if (lane == 0) {
            mbar_expect_tx(&bars[slot], 2 * bytes);
            bulk_g2s(ring + slot * kAttnSlot, a.k + off, bytes, &bars[slot], pol);
            bulk_g2s(ring + slot * kAttnSlot + kAttnUnitBytes, a.v + off, bytes, &bars[slot], pol);
        }
        ++ui;
    };
    int in_flight = 0;
    for (int i = 0; i < kAttnStages && ui < u1; ++i) {
        issue(i);
        ++in_flight;
    }
    // q, the partial records and the error word wait for the previous kernel on the stream
    griddep_wait();

    const float qscale = 1.4426950408889634f / sqrtf(static_cast<float>(kHeadDim));   // log2(e) / sqrt(d)
    float4 q4[MT];
    float mx[MT], ls[MT];
    float4 acc[MT];
    int head = -1, seg_idx = -1;
    bool dead = false;
    auto flush = [&]() {   // this warp's partial for `head` into record seg_idx
        if (head < 0) return;
        float* base = a.part + (static_cast<size_t>(z) * 2 + seg_idx) * a.M * kAttnRec;
#pragma unroll
        for (int m = 0; m < MT; ++m) {
            float* r = base + m * kAttnRec;
            *reinterpret_cast<float4*>(r + 4 * lane) = acc[m];
            if (lane == 0) {
                r[128] = mx[m];
                r[129] = ls[m];
            }
        }
    };
    int cslot = 0;
    uint32_t cphase = 0;
    int h = static_cast<int>(u0 / a.nch), c = static_cast<int>(u0 - static_cast<long long>(h) * a.nch) - 1;
    for (long long u = u0; u < u1; ++u) {
        if (++c == a.nch) {
            c = 0;
            ++h;
        }
        if (h != head) {
            flush();
            head = h;
            ++seg_idx;
#pragma unroll
            for (int m = 0; m < MT; ++m) {
                const float4 t = *reinterpret_cast<const float4*>(a.q + static_cast<size_t>(m) * a.q_stride + h * kHeadDim + 4 * lane);
                q4[m] = make_float4(t.x * qscale, t.y * qscale, t.z * qscale, t.w * qscale);
                mx[m] = -INFINITY;
                ls[m] = 0.0f;
                acc[m] = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
            }
        }
        if (!__all_sync(0xffffffffu, mbar_wait(&bars[cslot], cphase, a.wait_limit_ns))) {
            if (lane == 0) atomicCAS(a.err, 0, kDevErrTimeout);
            dead = true;   // cslot is the slot that timed out; in_flight counts it
            break;
        }
        attn_unit<MT>(smem_addr(ring + cslot * kAttnSlot) + 8 * lane, c * kAttnPos, min(kAttnPos, a.L - c * kAttnPos),
                      a.L - a.M, q4, mx, ls, acc, lane);
        __syncwarp();   // every lane's reads of the slot are done before it is refilled
        const int done_slot = cslot;
        cslot = (cslot + 1 == kAttnStages) ? 0 : cslot + 1;
        cphase ^= (cslot == 0) ? 1u : 0u;
        if (ui < u1) {
            issue(done_slot);
        } else {
            --in_flight;
        }
    }
    if (dead) {   // wait (bounded) for this warp's copies still in flight, then leave
        for (int j = 0; j < in_flight; ++j) {
            mbar_wait(&bars[cslot], cphase, a.wait_limit_ns);
            cslot = (cslot + 1 == kAttnStages) ? 0 : cslot + 1;
            cphase ^= (cslot == 0) ? 1u : 0u;
        }
    }
    flush();
}

// One CTA per (head, token): merges the partials of the warps whose units cover the head.  Warp w
// takes records w, w + 8, ... (lane l: dims [4l, 4l + 4)), loads them 8 at a time and combines them
// with a running maximum (each record's weighted sums rescaled by 2^(max_r - max)); warp 0 then
// combines the 8 warps' results in order, rescaled the same way: one round trip for the records, in
// a fixed order whatever the timing.
__global__ void __launch_bounds__(kThreads) aio_attn_combine_kernel(const __grid_constant__ AttnArgs a) {
    griddep_launch_dependents();
    __shared__ float4 wacc[kWarps][32];
    __shared__ float wml[kWarps][2];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int h = blockIdx.x / a.M, m = blockIdx.x - h * a.M;
    const long long ua = static_cast<long long>(h) * a.nch, ub = ua + a.nch - 1;   // the head's units
    long long zlo = ua * a.Z / a.U;   // the warp holding unit ua
    while (zlo > 0 && attn_seg(zlo, a.U, a.Z) > ua) --zlo;
    while (attn_seg(zlo + 1, a.U, a.Z) <= ua) ++zlo;
    long long zhi = ub * a.Z / a.U;   // the warp holding unit ub
    while (zhi > 0 && attn_seg(zhi, a.U, a.Z) > ub) --zhi;
    while (attn_seg(zhi + 1, a.U, a.Z) <= ub) ++zhi;
    const int n = static_cast<int>(zhi - zlo + 1);
    griddep_wait();   // the partial kernel has completed
    constexpr int B = 8;   // records a warp loads at once
    float gm = -INFINITY, gl = 0.0f;
    float4 acc = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
    for (int i0 = warp; i0 < n; i0 += B * kWarps) {
        float rm[B], rl[B];
        float4 rv[B];
#pragma unroll
        for (int b = 0; b < B; ++b) {   // the records' loads, issued together
            const int i = i0 + b * kWarps;
            rm[b] = -INFINITY;
            rl[b] = 0.0f;
            rv[b] = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
            if (i < n) {
                const long long zz = zlo + i, s0 = attn_seg(zz, a.U, a.Z);
                if (attn_seg(zz + 1, a.U, a.Z) > s0) {   // a non-empty segment: its first or second record
                    const float* r = a.part + ((zz * 2 + (s0 / a.nch == h ? 0 : 1)) * a.M + m) * kAttnRec;
                    rm[b] = r[128];
                    rl[b] = r[129];
                    rv[b] = *reinterpret_cast<const float4*>(r + 4 * lane);
                }
            }
        }
#pragma unroll
        for (int b = 0; b < B; ++b) {   // combined in record order
            if (rm[b] == -INFINITY) continue;
            const float nm = fmaxf(gm, rm[b]);
            const float so = exp2f(gm - nm), sr = exp2f(rm[b] - nm);   // so = 0 while gm is -inf
            gl = gl * so + rl[b] * sr;
            acc = make_float4(fmaf(rv[b].x, sr, acc.x * so), fmaf(rv[b].y, sr, acc.y * so), fmaf(rv[b].z, sr, acc.z * so),
                              fmaf(rv[b].w, sr, acc.w * so));
            gm = nm;
        }
    }
    wacc[warp][lane] = acc;
    if (lane == 0) {
        wml[warp][0] = gm;
        wml[warp][1] = gl;
    }
    __syncthreads();
    if (warp == 0) {
        float M_ = -INFINITY;
#pragma unroll
        for (int w = 0; w < kWarps; ++w) M_ = fmaxf(M_, wml[w][0]);
        float lt = 0.0f;
        float4 at = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
#pragma unroll
        for (int w = 0; w < kWarps; ++w) {
            const float sw = wml[w][0] == -INFINITY ? 0.0f : exp2f(wml[w][0] - M_);
            lt = fmaf(wml[w][1], sw, lt);
            const float4 v = wacc[w][lane];
            at = make_float4(fmaf(v.x, sw, at.x), fmaf(v.y, sw, at.y), fmaf(v.z, sw, at.z), fmaf(v.w, sw, at.w));
        }
        const float inv = 1.0f / lt;
        *reinterpret_cast<float4*>(a.out + static_cast<size_t>(m) * a.n_heads * kHeadDim + h * kHeadDim + 4 * lane) =
            make_float4(at.x * inv, at.y * inv, at.z * inv, at.w * inv);
    }
}

using AttnFn = void (*)(const AttnArgs);

AttnFn attn_fn(int M) {
    switch (M) {
        case 1: return aio_attn_partial_kernel<1>;
        case 2: return aio_attn_partial_kernel<2>;
        case 3: return aio_attn_partial_kernel<3>;
        case 4: return aio_attn_partial_kernel<4>;
        case 5: return aio_attn_partial_kernel<5>;
        case 6: return aio_attn_partial_kernel<6>;
        case 7: return aio_attn_partial_kernel<7>;
        case 8: return aio_attn_partial_kernel<8>;
        default: return nullptr;
    }
}

}  // namespace

size_t attn_workspace_bytes(int Z, int M) {
    return 256 + static_cast<size_t>(Z) * 2 * M * kAttnRec * sizeof(float);
}

cudaError_t launch_attention(const float* q, int q_stride, const void* k, const void* v, int n_heads, int L_max, int L,
                             int M, float* out, void* ws, int grid, unsigned long long wait_limit_ns, cudaStream_t s) {
    AttnFn f = attn_fn(M);
    if (!f) return cudaErrorInvalidValue;
    static thread_local int prepared_device = -1;
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (prepared_device != dev) {
        for (int i = 1; i <= kMaxM; ++i) {
            e = cudaFuncSetAttribute(attn_fn(i), cudaFuncAttributeMaxDynamicSharedMemorySize, kAttnSmem);
            if (e != cudaSuccess) return e;
        }
        prepared_device = dev;
    }
    AttnArgs a = {};
    a.q = q;
    a.k = static_cast<const uint16_t*>(k);
    a.v = static_cast<const uint16_t*>(v);
    a.out = out;
    a.err = static_cast<int*>(ws);
    a.part = reinterpret_cast<float*>(static_cast<uint8_t*>(ws) + 256);
    a.q_stride = q_stride;
    a.n_heads = n_heads;
    a.L_max = L_max;
    a.L = L;
    a.M = M;
    a.Z = grid * kWarps;
    a.nch = (L + kAttnPos - 1) / kAttnPos;
    a.U = static_cast<long long>(n_heads) * a.nch;
    a.wait_limit_ns = wait_limit_ns;
    // both with programmatic dependent launch (see the top of this file)
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr.val.programmaticStreamSerializationAllowed = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(grid));
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = kAttnSmem;
    cfg.stream = s;
    cfg.attrs = &attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, f, a);
    if (e != cudaSuccess) return e;
    cfg.gridDim = dim3(static_cast<unsigned>(n_heads * M));
    cfg.dynamicSmemBytes = 0;
    return cudaLaunchKernelEx(&cfg, aio_attn_combine_kernel, a);
}

}  // namespace aio
