// Weight Sum: out[t] = sum_j w[t,j] * y_pairs[pair_pos[t*k + j]] (+ y_shared[t]).
// One block per token gathers its k expert rows; fp32 sums in slot order,
// rounded once. No atomics, so the result does not depend on scheduling.
// A slot whose pair_pos is negative (a pair the permutation dropped) is
// skipped.
#include "common.cuh"
#include "kernels.h"

namespace gbmoe {

template <typename TA>
__global__ void __launch_bounds__(256)
combine_kernel(const TA* __restrict__ y, const float* __restrict__ w, const int32_t* __restrict__ pair_pos,
               const TA* __restrict__ y_shared, TA* __restrict__ out, int k, int H) {
    pdl_enter();
    const int t = blockIdx.x;
    __shared__ int32_t s_pos[32];
    __shared__ float s_w[32];
    if (threadIdx.x < k) {
        s_pos[threadIdx.x] = pair_pos[(size_t)t * k + threadIdx.x];
        s_w[threadIdx.x] = w[(size_t)t * k + threadIdx.x];
    }
    __syncthreads();
    for (int c = threadIdx.x; c < H / 8; c += blockDim.x) {
        float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
        for (int j = 0; j < k; ++j) {
            if (s_pos[j] < 0) continue;  // a dropped pair contributes nothing
            float v[8];
            Vec8<TA>::load(y + (size_t)s_pos[j] * H + 8 * c, v);
            const float wj = s_w[j];
#pragma unroll
            for (int i = 0; i < 8; ++i) acc[i] = __fmaf_rn(wj, v[i], acc[i]);
        }
        if (y_shared) {
            float v[8];
            Vec8<TA>::load(y_shared + (size_t)t * H + 8 * c, v);
#pragma unroll
            for (int i = 0; i < 8; ++i) acc[i] = __fadd_rn(acc[i], v[i]);
        }
        Vec8<TA>::store(out + (size_t)t * H + 8 * c, acc);
    }
}

cudaError_t launch_combine(const void* y_pairs, const float* topk_w, const int32_t* pair_pos, const void* y_shared,
                           void* out, int T, int k, int H, int act_dtype, cudaStream_t stream) {
    if (T == 0) return cudaSuccess;
    if (act_dtype == GBMOE_BF16)
        return launch_k(combine_kernel<__nv_bfloat16>, dim3(T), dim3(256), 0, stream,
                        static_cast<const __nv_bfloat16*>(y_pairs), topk_w, pair_pos,
                        static_cast<const __nv_bfloat16*>(y_shared), static_cast<__nv_bfloat16*>(out), k, H);
    return launch_k(combine_kernel<float>, dim3(T), dim3(256), 0, stream, static_cast<const float*>(y_pairs), topk_w,
                    pair_pos, static_cast<const float*>(y_shared), static_cast<float*>(out), k, H);
}

}  // namespace gbmoe
