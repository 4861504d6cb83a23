// Streaming FFN kernels instantiated for GBMOE_F32 expert weights.
#include "ffn_stream.cuh"

namespace gbmoe {

template <>
cudaError_t launch_stream_w<GBMOE_F32>(const FfnProblem& p, cudaStream_t stream) {
    return launch_stream_t<float, GBMOE_F32>(p, stream);
}

}  // namespace gbmoe
