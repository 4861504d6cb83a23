// Streaming FFN route: shared-memory size of a CTA and the dispatch over
// weight formats (the kernels are in ffn_stream.cuh, instantiated per format
// in ffn_stream_<format>.cu).
#include "ffn_stream.cuh"

namespace gbmoe {

size_t stream_smem_bytes(int act_dtype, int H, int I) {
    const size_t ab = act_dtype == GBMOE_F32 ? 4 : 2;
    const size_t a = (size_t)kNT * H * ab, b = (size_t)kNT * I * ab;
    return a > b ? a : b;
}

cudaError_t launch_ffn_stream(const FfnProblem& p, cudaStream_t stream) {
    cudaError_t err = launch_ffn_schedule(p.counts, p.E, p.n_rows, kSchedMinBM, p.sched, stream);
    if (err != cudaSuccess) return err;
    switch (p.w_dtype) {
        case GBMOE_F32: return p.act_dtype == GBMOE_F32 ? launch_stream_w<GBMOE_F32>(p, stream) : cudaErrorInvalidValue;
        case GBMOE_BF16: return launch_stream_w<GBMOE_BF16>(p, stream);
        case GBMOE_FP8_E4M3_B128: return launch_stream_w<GBMOE_FP8_E4M3_B128>(p, stream);
        case GBMOE_INT4_G128: return launch_stream_w<GBMOE_INT4_G128>(p, stream);
        case GBMOE_MXFP4: return launch_stream_w<GBMOE_MXFP4>(p, stream);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace gbmoe
