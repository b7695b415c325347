// aio_chain_ph.cu -- instantiates the stream kernel for chained steps that also have attention,
// merge or SwiGLU phases (attention over a KV cache before O; a SwiGLU x too large to stage),
// M <= kMaxChainM.
#include "aio_stream.cuh"

namespace aio {

StreamFn chain_phase_stream_fn(bool i8, int M) {
    switch (M) {
        case 1: return i8 ? aio_stream_kernel<1, true, true, true> : aio_stream_kernel<1, false, true, true>;
        case 2: return i8 ? aio_stream_kernel<2, true, true, true> : aio_stream_kernel<2, false, true, true>;
        case 3: return i8 ? aio_stream_kernel<3, true, true, true> : aio_stream_kernel<3, false, true, true>;
        case 4: return i8 ? aio_stream_kernel<4, true, true, true> : aio_stream_kernel<4, false, true, true>;
        default: return nullptr;
    }
}

}  // namespace aio
