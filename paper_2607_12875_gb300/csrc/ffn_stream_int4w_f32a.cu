// Streaming FFN kernels instantiated for GBMOE_INT4_G128 expert weights with
// fp32 activations.
#include "ffn_stream.cuh"

namespace gbmoe {

cudaError_t launch_stream_int4w_f32a(const FfnProblem& p, cudaStream_t stream) {
    return launch_stream_t<float, GBMOE_INT4_G128>(p, stream);
}

}  // namespace gbmoe
