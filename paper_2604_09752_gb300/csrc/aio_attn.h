// Declarations of the decode-attention launcher (aio_attn.cu) for the C ABI (aio_api.cu); not part
// of the ABI.
#pragma once

#include "aio_internal.h"

namespace aio {

// Workspace bytes for Z warps and M tokens: a 256-byte header (the device error word), then the
// per-warp partial results.
size_t attn_workspace_bytes(int Z, int M);

// The partial kernel over `grid` CTAs, then the merge kernel, on stream s.
cudaError_t launch_attention(const float* q, int q_stride, const void* k, const void* v, int n_heads, int L_max, int L,
                             int M, float* out, void* ws, int grid, unsigned long long wait_limit_ns, cudaStream_t s);

}  // namespace aio
