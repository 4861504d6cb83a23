// Streaming FFN kernels instantiated for GBMOE_FP8_E4M3_B128 expert weights.
#include "ffn_stream.cuh"

namespace gbmoe {

template <>
cudaError_t launch_stream_w<GBMOE_FP8_E4M3_B128>(const FfnProblem& p, cudaStream_t stream) {
    return p.act_dtype == GBMOE_BF16 ? launch_stream_t<__nv_bfloat16, GBMOE_FP8_E4M3_B128>(p, stream)
                                     : launch_stream_t<float, GBMOE_FP8_E4M3_B128>(p, stream);
}

}  // namespace gbmoe
