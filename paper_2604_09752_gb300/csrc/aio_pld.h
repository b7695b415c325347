// Declarations of the prompt-lookup launchers (aio_pld.cu) for the C ABI (aio_api.cu); not part of
// the ABI.
#pragma once

#include <cuda_runtime.h>

namespace aio {

constexpr int kPldMaxN = 32;   // longest n-gram window
constexpr int kPldMaxL = 7;    // longest look-ahead (the verification pass then has <= 8 rows)

cudaError_t launch_pld_draft(const int* tokens, int T, int N, int L, int* out, cudaStream_t s);
cudaError_t launch_argmax(const float* logits, int M, int V, int stride, int* out, cudaStream_t s);
cudaError_t launch_pld_accept(const int* argmax, const int* draft, int* result, cudaStream_t s);
cudaError_t launch_route(const float* logits, const int* cat_tok, int n, int code, int L_ctx, float tau, int* decision,
                         cudaStream_t s);

}  // namespace aio
