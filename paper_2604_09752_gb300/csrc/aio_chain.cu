// aio_chain.cu -- instantiates the stream kernel for chained steps (a projection's x may be
// computed on the device: RMSNorm with a residual add, SwiGLU, a column slice), M <= kMaxChainM.
#include "aio_stream.cuh"

namespace aio {

StreamFn chain_stream_fn(bool i8, int M, bool phases) {
    if (phases) return chain_phase_stream_fn(i8, M);
    switch (M) {
        case 1: return i8 ? aio_stream_kernel<1, true, true> : aio_stream_kernel<1, false, true>;
        case 2: return i8 ? aio_stream_kernel<2, true, true> : aio_stream_kernel<2, false, true>;
        case 3: return i8 ? aio_stream_kernel<3, true, true> : aio_stream_kernel<3, false, true>;
        case 4: return i8 ? aio_stream_kernel<4, true, true> : aio_stream_kernel<4, false, true>;
        default: return nullptr;
    }
}

}  // namespace aio
