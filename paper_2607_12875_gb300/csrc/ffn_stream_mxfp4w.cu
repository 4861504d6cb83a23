// Streaming FFN kernels instantiated for GBMOE_MXFP4 expert weights.
#include "ffn_stream.cuh"

namespace gbmoe {

template <>
cudaError_t launch_stream_w<GBMOE_MXFP4>(const FfnProblem& p, cudaStream_t stream) {
    return p.act_dtype == GBMOE_BF16 ? launch_stream_t<__nv_bfloat16, GBMOE_MXFP4>(p, stream)
                                     : launch_stream_t<float, GBMOE_MXFP4>(p, stream);
}

}  // namespace gbmoe
