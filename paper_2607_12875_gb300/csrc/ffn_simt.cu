// Fused MoE on CUDA cores: tiled grouped GEMMs in fp32.
//
// The route for fp32 activations (where tensor-core inputs would lose the
// fp32 precision the layer is specified in) and for any weight format. A CTA
// computes a 32x32 output tile of one expert's rows: stage 1 produces both
// the gate and the up tile and writes h = silu(g) * u, stage 2 multiplies h by
// the expert's down matrix. Weights are decoded to fp32 as they are staged.
#include "common.cuh"
#include "ffn_sched.h"
#include "kernels.h"
#include "wload.cuh"

namespace gbmoe {

constexpr int kBM = 32, kBN = 32, kBK = 32;
static_assert(kBM == kSchedMinBM, "tile list is built for the SIMT tile height");

template <typename TA, int WQ>
__global__ void __launch_bounds__(256)
simt_gateup_kernel(FfnProblem p) {
    pdl_enter();
    __shared__ float As[kBM][kBK + 1];
    __shared__ float Bg[kBN][kBK + 1];
    __shared__ float Bu[kBN][kBK + 1];
    __shared__ int32_t s_src[kBM];
    const int32_t* sched = p.sched;
    const int tile = blockIdx.x;
    if (tile >= sched[1]) return;
    const int2 tl = reinterpret_cast<const int2*>(sched + sched_tiles_offset(p.E))[tile];
    const int e = tl.x;
    const int64_t cnt = p.counts ? p.counts[e] : p.n_rows;
    const int64_t row0 = (p.offsets ? p.offsets[e] : 0) + (int64_t)tl.y * kBM;
    const int rows = (int)min64(kBM, cnt - (int64_t)tl.y * kBM);
    const int i0 = blockIdx.y * kBN;
    const int H = p.H, I = p.I;
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    if (threadIdx.x < kBM) {
        int64_t r = row0 + threadIdx.x;
        s_src[threadIdx.x] = threadIdx.x < rows ? (p.sorted_pair ? p.sorted_pair[r] / p.pair_div : (int32_t)r) : -1;
    }
    __syncthreads();
    const TA* x = static_cast<const TA*>(p.x);
    float ag[2][2] = {{0.f, 0.f}, {0.f, 0.f}}, au[2][2] = {{0.f, 0.f}, {0.f, 0.f}};
    for (int k0 = 0; k0 < H; k0 += kBK) {
        for (int idx = threadIdx.x; idx < kBM * kBK; idx += 256) {
            int r = idx / kBK, kk = idx % kBK;
            int src = s_src[r];
            As[r][kk] = src >= 0 ? to_f32(x[(size_t)src * H + k0 + kk]) : 0.0f;
            Bg[r][kk] = WFmt<WQ>::elem(p.w_gate, p.s_gate, e, I, H, i0 + r, k0 + kk);
            Bu[r][kk] = WFmt<WQ>::elem(p.w_up, p.s_up, e, I, H, i0 + r, k0 + kk);
        }
        __syncthreads();
#pragma unroll 8
        for (int kk = 0; kk < kBK; ++kk) {
            float a0 = As[ty * 2][kk], a1 = As[ty * 2 + 1][kk];
            float g0 = Bg[tx * 2][kk], g1 = Bg[tx * 2 + 1][kk];
            float u0 = Bu[tx * 2][kk], u1 = Bu[tx * 2 + 1][kk];
            ag[0][0] = fmaf(a0, g0, ag[0][0]); ag[0][1] = fmaf(a0, g1, ag[0][1]);
            ag[1][0] = fmaf(a1, g0, ag[1][0]); ag[1][1] = fmaf(a1, g1, ag[1][1]);
            au[0][0] = fmaf(a0, u0, au[0][0]); au[0][1] = fmaf(a0, u1, au[0][1]);
            au[1][0] = fmaf(a1, u0, au[1][0]); au[1][1] = fmaf(a1, u1, au[1][1]);
        }
        __syncthreads();
    }
    TA* h = static_cast<TA*>(p.h);
#pragma unroll
    for (int a = 0; a < 2; ++a) {
        int r = ty * 2 + a;
        if (r >= rows) continue;
#pragma unroll
        for (int b = 0; b < 2; ++b) h[(row0 + r) * I + i0 + tx * 2 + b] = from_f32<TA>(silu_mul(ag[a][b], au[a][b]));
    }
}

template <typename TA, int WQ>
__global__ void __launch_bounds__(256)
simt_down_kernel(FfnProblem p) {
    pdl_enter();
    __shared__ float As[kBM][kBK + 1];
    __shared__ float Bd[kBN][kBK + 1];
    const int32_t* sched = p.sched;
    const int tile = blockIdx.x;
    if (tile >= sched[1]) return;
    const int2 tl = reinterpret_cast<const int2*>(sched + sched_tiles_offset(p.E))[tile];
    const int e = tl.x;
    const int64_t cnt = p.counts ? p.counts[e] : p.n_rows;
    const int64_t row0 = (p.offsets ? p.offsets[e] : 0) + (int64_t)tl.y * kBM;
    const int rows = (int)min64(kBM, cnt - (int64_t)tl.y * kBM);
    const int n0 = blockIdx.y * kBN;
    const int H = p.H, I = p.I;
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    const TA* h = static_cast<const TA*>(p.h);
    float acc[2][2] = {{0.f, 0.f}, {0.f, 0.f}};
    for (int k0 = 0; k0 < I; k0 += kBK) {
        for (int idx = threadIdx.x; idx < kBM * kBK; idx += 256) {
            int r = idx / kBK, kk = idx % kBK;
            As[r][kk] = r < rows ? to_f32(h[(row0 + r) * I + k0 + kk]) : 0.0f;
            Bd[r][kk] = WFmt<WQ>::elem(p.w_down, p.s_down, e, H, I, n0 + r, k0 + kk);
        }
        __syncthreads();
#pragma unroll 8
        for (int kk = 0; kk < kBK; ++kk) {
            float a0 = As[ty * 2][kk], a1 = As[ty * 2 + 1][kk];
            float b0 = Bd[tx * 2][kk], b1 = Bd[tx * 2 + 1][kk];
            acc[0][0] = fmaf(a0, b0, acc[0][0]); acc[0][1] = fmaf(a0, b1, acc[0][1]);
            acc[1][0] = fmaf(a1, b0, acc[1][0]); acc[1][1] = fmaf(a1, b1, acc[1][1]);
        }
        __syncthreads();
    }
    TA* y = static_cast<TA*>(p.y);
#pragma unroll
    for (int a = 0; a < 2; ++a) {
        int r = ty * 2 + a;
        if (r >= rows) continue;
#pragma unroll
        for (int b = 0; b < 2; ++b) y[(row0 + r) * H + n0 + tx * 2 + b] = from_f32<TA>(acc[a][b]);
    }
}

template <typename TA, int WQ>
static cudaError_t launch_simt_t(const FfnProblem& p, cudaStream_t stream) {
    const int64_t max_tiles = sched_max_tiles(p.E, p.n_rows, kBM);
    if (p.n_rows == 0) return cudaSuccess;
    dim3 g1((unsigned)max_tiles, p.I / kBN);
    if (const cudaError_t le = launch_k(simt_gateup_kernel<TA, WQ>, dim3(g1), dim3(256), 0, stream, p); le != cudaSuccess)
        return le;
    cudaError_t err = cudaGetLastError();
    if (err != cudaSuccess) return err;
    dim3 g2((unsigned)max_tiles, p.H / kBN);
    if (const cudaError_t le = launch_k(simt_down_kernel<TA, WQ>, dim3(g2), dim3(256), 0, stream, p); le != cudaSuccess)
        return le;
    return cudaGetLastError();
}

cudaError_t launch_ffn_simt(const FfnProblem& p, cudaStream_t stream) {
    cudaError_t err = launch_ffn_schedule(p.counts, p.E, p.n_rows, kBM, p.sched, stream);
    if (err != cudaSuccess) return err;
    if (p.act_dtype == GBMOE_BF16) {
        switch (p.w_dtype) {
            case GBMOE_F32: return launch_simt_t<__nv_bfloat16, GBMOE_F32>(p, stream);
            case GBMOE_BF16: return launch_simt_t<__nv_bfloat16, GBMOE_BF16>(p, stream);
            case GBMOE_FP8_E4M3_B128: return launch_simt_t<__nv_bfloat16, GBMOE_FP8_E4M3_B128>(p, stream);
            case GBMOE_INT4_G128: return launch_simt_t<__nv_bfloat16, GBMOE_INT4_G128>(p, stream);
            case GBMOE_MXFP4: return launch_simt_t<__nv_bfloat16, GBMOE_MXFP4>(p, stream);
            default: return cudaErrorInvalidValue;
        }
    }
    switch (p.w_dtype) {
        case GBMOE_F32: return launch_simt_t<float, GBMOE_F32>(p, stream);
        case GBMOE_BF16: return launch_simt_t<float, GBMOE_BF16>(p, stream);
        case GBMOE_FP8_E4M3_B128: return launch_simt_t<float, GBMOE_FP8_E4M3_B128>(p, stream);
        case GBMOE_INT4_G128: return launch_simt_t<float, GBMOE_INT4_G128>(p, stream);
        case GBMOE_MXFP4: return launch_simt_t<float, GBMOE_MXFP4>(p, stream);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace gbmoe
