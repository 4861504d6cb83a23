// Streaming FFN kernels instantiated for GBMOE_INT4_G128 expert weights with
// bf16 activations (fp32 activations: ffn_stream_int4w_f32a.cu).
#include "ffn_stream.cuh"

namespace gbmoe {

template <>
cudaError_t launch_stream_w<GBMOE_INT4_G128>(const FfnProblem& p, cudaStream_t stream) {
    return p.act_dtype == GBMOE_BF16 ? launch_stream_t<__nv_bfloat16, GBMOE_INT4_G128>(p, stream)
                                     : launch_stream_int4w_f32a(p, stream);
}

}  // namespace gbmoe
