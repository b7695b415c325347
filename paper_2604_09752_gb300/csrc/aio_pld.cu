// aio_pld.cu -- prompt-lookup decoding around the verification pass (Sec. 4.2: n-gram matching
// window N = 6, look-ahead L = 2), and the routing decision.  Small kernels, mostly integer or
// comparison work:
//   * draft:  among positions i < T - 1, the one whose preceding tokens share the longest suffix
//             (<= N) with the whole sequence, the most recent among equals; the draft is the up to
//             L tokens after it.  One CTA: every thread scores positions i = tid, tid + 1024, ...
//             (at most N comparisons each) and a block reduction picks max (n, i).
//   * argmax: one CTA per row of logits; ties go to the lowest index, NaN counts as the maximum
//             (the first NaN wins), as numpy's argmax does.
//   * accept: greedy acceptance of the drafted tokens against the verification pass's argmax.
//   * route:  the request-level decision of Sec. 3.2 and Sec. 3.3 from the probe's logits over the
//             category tokens: category (argmax), softmax entropy in nats against tau, the model
//             (1B only for confident Code Generation with L_ctx <= 2048) and the PLD switch.
#include <cuda_runtime.h>
#include <stdint.h>

#include "aio_pld.h"

namespace aio {
namespace {

constexpr int kPldThreads = 1024;

// Larger key wins: longer match first, then the more recent position.
__device__ __forceinline__ unsigned long long pld_key(int n, int i) {
    return (static_cast<unsigned long long>(n) << 32) | static_cast<unsigned>(i);
}

__global__ void __launch_bounds__(kPldThreads) aio_pld_draft_kernel(const int* __restrict__ tok, int T, int N, int L,
                                                                    int* __restrict__ out) {
    __shared__ int suf[kPldMaxN];
    __shared__ unsigned long long wbest[kPldThreads / 32];
    if (threadIdx.x < N) suf[threadIdx.x] = threadIdx.x < T ? tok[T - 1 - threadIdx.x] : 0;
    __syncthreads();
    unsigned long long best = 0;   // n = 0: no match
    for (int i = threadIdx.x; i < T - 1; i += kPldThreads) {
        int n = 0;
        while (n < N && i - n >= 0 && tok[i - n] == suf[n]) ++n;
        if (n > 0) {
            const unsigned long long k = pld_key(n, i);
            best = k > best ? k : best;
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const unsigned long long other = __shfl_xor_sync(0xffffffffu, best, o);
        best = other > best ? other : best;
    }
    if ((threadIdx.x & 31) == 0) wbest[threadIdx.x >> 5] = best;
    __syncthreads();
    if (threadIdx.x == 0) {
        unsigned long long b = 0;
        for (int w = 0; w < kPldThreads / 32; ++w) b = wbest[w] > b ? wbest[w] : b;
        const int n = static_cast<int>(b >> 32);
        const int i = n ? static_cast<int>(b & 0xFFFFFFFFu) : -1;
        const int d = n ? min(L, T - 1 - i) : 0;
        out[0] = d;
        out[1] = n;
        out[2] = i;
        for (int j = 0; j < L; ++j) out[3 + j] = j < d ? tok[i + 1 + j] : -1;
    }
}

// a better than b (with indices ia, ib): NaN above every number, then larger, then lower index.
__device__ __forceinline__ bool argmax_better(float a, int ia, float b, int ib) {
    const bool na = a != a, nb = b != b;
    if (na != nb) return na;
    if (!na && a != b) return a > b;
    return ia < ib;
}

__global__ void __launch_bounds__(kPldThreads) aio_argmax_kernel(const float* __restrict__ logits, int V, int stride,
                                                                 int* __restrict__ out) {
    __shared__ float wv[kPldThreads / 32];
    __shared__ int wi[kPldThreads / 32];
    const float* row = logits + static_cast<size_t>(blockIdx.x) * stride;
    float bv = 0.0f;
    int bi = -1;
    for (int j = threadIdx.x; j < V; j += kPldThreads) {
        const float v = row[j];
        if (bi < 0 || argmax_better(v, j, bv, bi)) {
            bv = v;
            bi = j;
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
        const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
        if (oi >= 0 && (bi < 0 || argmax_better(ov, oi, bv, bi))) {
            bv = ov;
            bi = oi;
        }
    }
    if ((threadIdx.x & 31) == 0) {
        wv[threadIdx.x >> 5] = bv;
        wi[threadIdx.x >> 5] = bi;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        float v = wv[0];
        int i = wi[0];
        for (int w = 1; w < kPldThreads / 32; ++w)
            if (wi[w] >= 0 && (i < 0 || argmax_better(wv[w], wi[w], v, i))) {
                v = wv[w];
                i = wi[w];
            }
        out[blockIdx.x] = i;
    }
}

__global__ void aio_pld_accept_kernel(const int* __restrict__ argmax, const int* __restrict__ draft,
                                      int* __restrict__ result) {
    const int d = draft[0];
    int a = 0;
    while (a < d && argmax[a] == draft[3 + a]) ++a;
    result[0] = a;
    result[1] = argmax[a];
}

// One warp; lane c < n holds category c.
__global__ void aio_route_kernel(const float* __restrict__ logits, const int* __restrict__ cat_tok, int n, int code,
                                 int L_ctx, float tau, int* __restrict__ decision) {
    const int lane = threadIdx.x;
    const float l = lane < n ? logits[cat_tok[lane]] : -INFINITY;
    float mx = l;
    int arg = lane < n ? lane : 0x7FFFFFFF;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float om = __shfl_xor_sync(0xffffffffu, mx, o);
        const int oa = __shfl_xor_sync(0xffffffffu, arg, o);
        if (om > mx || (om == mx && oa < arg)) {
            mx = om;
            arg = oa;
        }
    }
    const float e = lane < n ? expf(l - mx) : 0.0f;
    float sum = e;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
    const float p = e / sum;
    float t = p > 0.0f ? p * logf(p) : 0.0f;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
    const float H = -t;
    if (lane == 0) {
        const bool is_code = arg == code;
        decision[0] = arg;
        decision[1] = (is_code && L_ctx <= 2048 && H <= tau) ? 1 : 7;
        decision[2] = is_code ? 0 : 1;
        decision[3] = __float_as_int(H);
    }
}

}  // namespace

cudaError_t launch_route(const float* logits, const int* cat_tok, int n, int code, int L_ctx, float tau, int* decision,
                         cudaStream_t s) {
    aio_route_kernel<<<1, 32, 0, s>>>(logits, cat_tok, n, code, L_ctx, tau, decision);
    return cudaGetLastError();
}

cudaError_t launch_pld_draft(const int* tokens, int T, int N, int L, int* out, cudaStream_t s) {
    aio_pld_draft_kernel<<<1, kPldThreads, 0, s>>>(tokens, T, N, L, out);
    return cudaGetLastError();
}

cudaError_t launch_argmax(const float* logits, int M, int V, int stride, int* out, cudaStream_t s) {
    aio_argmax_kernel<<<M, kPldThreads, 0, s>>>(logits, V, stride, out);
    return cudaGetLastError();
}

cudaError_t launch_pld_accept(const int* argmax, const int* draft, int* result, cudaStream_t s) {
    aio_pld_accept_kernel<<<1, 1, 0, s>>>(argmax, draft, result);
    return cudaGetLastError();
}

}  // namespace aio
