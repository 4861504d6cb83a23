// Fused MoE for few rows per expert (decode): weight streaming.
//
// With ~2 rows per expert the layer is bound by reading each active expert's
// weights once from HBM. Each CTA takes one active expert and a slice of
// output columns; its warps stream weight rows with 16-byte non-allocating
// loads (kUnroll chunks of each of its 4 rows in flight per lane: 8 KB per
// warp) and dot them against the expert's activation rows, which sit in
// shared memory. Lane l takes the 16-byte chunks l, l+32, ... of a row, so a
// warp reads 512 contiguous bytes per row and step. The inner loop reloads
// each activation chunk once and decodes the weights per activation row, so
// the kernel stays within 128 registers and two CTAs (16 warps) share an SM.
// Up to kNT rows are handled per weight pass; more rows take further passes
// over the same weights. A CTA covers up to 4 column groups in turn, so it
// stages its activation rows once for all of them.
//   stage 1: h[r, i] = silu(x_r . Wgate[i]) * (x_r . Wup[i]), 2 columns per warp
//   stage 2: y[r, n] = h_r . Wdown[n], 4 output columns per warp
#pragma once

#include <type_traits>

#include "common.cuh"
#include "ffn_sched.h"
#include "kernels.h"
#include "wload.cuh"

namespace gbmoe {

constexpr int kStreamWarps = 8;
constexpr int kNT = 8;      // activation rows per weight pass
constexpr int kUnroll = 4;  // chunks per row loaded before use
constexpr int kMaxGroupsPerCta = 4;
constexpr int kMinWaves = 8;

// CTAs per SM the register budget is set for: two for bf16 weights (the
// decode path); fp32 and quantised weights hold or decode more per element
// and get the whole register file
template <int WQ>
constexpr int stream_min_blocks() { return WQ == GBMOE_BF16 ? 2 : 1; }

// acc[q][r] += W_q . xs[r] for 4 weight rows q (byte pointers wrow, scale rows
// srow) and NT activation rows r in shared memory (row stride K).
template <typename TA, int WQ, int NT>
__device__ __forceinline__ void dot4(const uint8_t* const (&wrow)[4], const void* const (&srow)[4], const TA* xs,
                                     int K, float (&acc)[4][NT]) {
    using F = WFmt<WQ>;
    const int lane = threadIdx.x & 31;
    const int nchunk = K / F::CE;
    constexpr int CB = F::NV * 16;  // bytes per chunk
    for (int c0 = lane; c0 < nchunk; c0 += 32 * kUnroll) {
        uint4 raw[kUnroll][4][F::NV];
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
            const int c = c0 + 32 * u;
#pragma unroll
            for (int q = 0; q < 4; ++q)
#pragma unroll
                for (int v = 0; v < F::NV; ++v)
                    raw[u][q][v] = c < nchunk ? ld_stream16(wrow[q] + (size_t)c * CB + 16 * v) : make_uint4(0, 0, 0, 0);
        }
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
            const int c = c0 + 32 * u;
            if (c >= nchunk) break;
            float sc[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) sc[q] = F::scale_at(srow[q], c * F::CE);
#pragma unroll
            for (int sub = 0; sub < F::CE / 8; ++sub) {
                const int k0 = c * F::CE + 8 * sub;
#pragma unroll
                for (int r = 0; r < NT; ++r) {
                    float xv[8];
                    Vec8<TA>::load(xs + (size_t)r * K + k0, xv);
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        float w[8];
                        F::decode8(raw[u][q], sub, sc[q], w);
#pragma unroll
                        for (int i = 0; i < 8; ++i) acc[q][r] = fmaf(w[i], xv[i], acc[q][r]);
                    }
                }
            }
        }
    }
}

template <int NT>
__device__ __forceinline__ void warp_sum(float (&acc)[4][NT]) {
#pragma unroll
    for (int q = 0; q < 4; ++q)
#pragma unroll
        for (int r = 0; r < NT; ++r) {
            float v = acc[q][r];
#pragma unroll
            for (int d = 16; d >= 1; d >>= 1) v += __shfl_xor_sync(0xffffffffu, v, d);
            acc[q][r] = v;
        }
}

// Copies nt activation rows into shared memory: row r is source row
// sorted_pair[row0 + r] / pair_div (row0 + r itself without sorted_pair).
template <typename TA>
__device__ void stage_rows(TA* xs, const TA* src, int K, const int32_t* sorted_pair, int pair_div, int64_t row0,
                           int nt) {
    const int per_row = K * (int)sizeof(TA) / 16;
    for (int idx = threadIdx.x; idx < nt * per_row; idx += blockDim.x) {
        const int r = idx / per_row, c = idx % per_row;
        int64_t srow = row0 + r;
        if (sorted_pair) srow = sorted_pair[srow] / pair_div;
        reinterpret_cast<uint4*>(xs + (size_t)r * K)[c] = reinterpret_cast<const uint4*>(src + srow * K)[c];
    }
}

template <typename F>
__device__ __forceinline__ void dispatch_nt(int nt, F&& f) {
    if (nt <= 1) f(std::integral_constant<int, 1>{});
    else if (nt <= 2) f(std::integral_constant<int, 2>{});
    else if (nt <= 4) f(std::integral_constant<int, 4>{});
    else f(std::integral_constant<int, 8>{});
}

// Weight rows of column group g: 2 gate + 2 up rows (stage 1) or 4 down rows
// (stage 2) per warp, with their scale rows; col0 = first output column.
template <int WQ, int STAGE>
__device__ __forceinline__ void group_rows(const FfnProblem& p, int e, int g, int warp, const uint8_t* (&wrow)[4],
                                           const void* (&srow)[4], int& col0) {
    using F = WFmt<WQ>;
    const int H = p.H, I = p.I;
    if (STAGE == 1) {
        const size_t rb = F::row_bytes(H);
        const int i0 = (g * kStreamWarps + warp) * 2;
        const uint8_t* wg = static_cast<const uint8_t*>(p.w_gate) + (size_t)e * I * rb;
        const uint8_t* wu = static_cast<const uint8_t*>(p.w_up) + (size_t)e * I * rb;
        wrow[0] = wg + i0 * rb; wrow[1] = wg + (i0 + 1) * rb; wrow[2] = wu + i0 * rb; wrow[3] = wu + (i0 + 1) * rb;
        srow[0] = F::scale_row(p.s_gate, e, I, H, i0); srow[1] = F::scale_row(p.s_gate, e, I, H, i0 + 1);
        srow[2] = F::scale_row(p.s_up, e, I, H, i0); srow[3] = F::scale_row(p.s_up, e, I, H, i0 + 1);
        col0 = i0;
    } else {
        const size_t rb = F::row_bytes(I);
        const int n0 = (g * kStreamWarps + warp) * 4;
        const uint8_t* wd = static_cast<const uint8_t*>(p.w_down) + (size_t)e * H * rb;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            wrow[q] = wd + (n0 + q) * rb;
            srow[q] = F::scale_row(p.s_down, e, H, I, n0 + q);
        }
        col0 = n0;
    }
}

// One CTA: one active expert and gpc consecutive column groups (a group is 8
// warps x 2 h-columns in stage 1, 8 warps x 4 y-columns in stage 2). The
// expert's activation rows are staged once per pass of kNT rows and serve
// all of the CTA's groups.
//   stage 1: h[r, i] = silu(x_r . Wgate[i]) * (x_r . Wup[i])
//   stage 2: y[r, n] = h_r . Wdown[n]
template <typename TA, int WQ, int STAGE>
__device__ __forceinline__ void stream_ffn_cta(const FfnProblem& p, int gpc) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    TA* xs = reinterpret_cast<TA*>(smem_raw);
    const int slot = blockIdx.x;
    if (slot >= p.sched[0]) return;
    const int e = p.sched[kSchedHeader + slot];
    const int64_t cnt = p.counts ? p.counts[e] : p.n_rows;
    const int64_t row0 = p.offsets ? p.offsets[e] : 0;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int K = STAGE == 1 ? p.H : p.I;
    TA* out = static_cast<TA*>(STAGE == 1 ? p.h : p.y);
    const int out_cols = STAGE == 1 ? p.I : p.H;
    for (int64_t p0 = 0; p0 < cnt; p0 += kNT) {
        const int nt = (int)min64(kNT, cnt - p0);
        __syncthreads();
        if (STAGE == 1) stage_rows<TA>(xs, static_cast<const TA*>(p.x), K, p.sorted_pair, p.pair_div, row0 + p0, nt);
        else stage_rows<TA>(xs, static_cast<const TA*>(p.h), K, nullptr, 1, row0 + p0, nt);
        __syncthreads();
        dispatch_nt(nt, [&](auto NTc) {
            constexpr int NT = decltype(NTc)::value;
#pragma unroll 1
            for (int g = blockIdx.y * gpc; g < (blockIdx.y + 1) * gpc; ++g) {
                const uint8_t* wrow[4];
                const void* srow[4];
                int col0;
                group_rows<WQ, STAGE>(p, e, g, warp, wrow, srow, col0);
                float acc[4][NT];
#pragma unroll
                for (int q = 0; q < 4; ++q)
#pragma unroll
                    for (int r = 0; r < NT; ++r) acc[q][r] = 0.0f;
                dot4<TA, WQ, NT>(wrow, srow, xs, K, acc);
                warp_sum<NT>(acc);
#pragma unroll
                for (int r = 0; r < NT; ++r)
                    if (r == lane && r < nt) {
                        TA* dst = out + (row0 + p0 + r) * out_cols + col0;
                        if (STAGE == 1) {
                            dst[0] = from_f32<TA>(silu_mul(acc[0][r], acc[2][r]));
                            dst[1] = from_f32<TA>(silu_mul(acc[1][r], acc[3][r]));
                        } else {
#pragma unroll
                            for (int q = 0; q < 4; ++q) dst[q] = from_f32<TA>(acc[q][r]);
                        }
                    }
            }
        });
    }
}

template <typename TA, int WQ>
__global__ void __launch_bounds__(kStreamWarps * 32, stream_min_blocks<WQ>())
stream_gateup_kernel(FfnProblem p, int gpc) {
    pdl_enter();
    stream_ffn_cta<TA, WQ, 1>(p, gpc);
}

template <typename TA, int WQ>
__global__ void __launch_bounds__(kStreamWarps * 32, stream_min_blocks<WQ>())
stream_down_kernel(FfnProblem p, int gpc) {
    pdl_enter();
    stream_ffn_cta<TA, WQ, 2>(p, gpc);
}

// Column groups per CTA: up to kMaxGroupsPerCta while the grid keeps at least
// kMinWaves waves of CTAs (fewer, longer CTAs stage the rows less often;
// too few CTAs leave SMs idle). groups is a multiple of 8.
inline int groups_per_cta(int max_active, int groups) {
    const int64_t slots = (int64_t)sm_count() * 2;  // resident CTAs (two per SM)
    int gpc = kMaxGroupsPerCta;
    while (gpc > 1 && (int64_t)max_active * (groups / gpc) < kMinWaves * slots) gpc /= 2;
    return gpc;
}

template <typename TA, int WQ>
static cudaError_t launch_stream_t(const FfnProblem& p, cudaStream_t stream) {
    const int max_active = (int)min64(p.E, p.n_rows);
    if (max_active == 0) return cudaSuccess;
    const size_t smem1 = (size_t)kNT * p.H * sizeof(TA);
    const size_t smem2 = (size_t)kNT * p.I * sizeof(TA);
    cudaError_t err;
    // the largest dynamic shared memory any problem may ask for, set once per device
    static DeviceOnce smem_set;
    err = smem_set.run([] {
        const int most = (int)stream_smem_budget();
        cudaError_t e = cudaFuncSetAttribute(stream_gateup_kernel<TA, WQ>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, most);
        if (e != cudaSuccess) return e;
        return cudaFuncSetAttribute(stream_down_kernel<TA, WQ>, cudaFuncAttributeMaxDynamicSharedMemorySize, most);
    });
    if (err != cudaSuccess) return err;
    const int groups1 = p.I / (2 * kStreamWarps), groups2 = p.H / (4 * kStreamWarps);
    const int gpc1 = groups_per_cta(max_active, groups1), gpc2 = groups_per_cta(max_active, groups2);
    dim3 g1(max_active, groups1 / gpc1);
    if (const cudaError_t le = launch_k(stream_gateup_kernel<TA, WQ>, dim3(g1), dim3(kStreamWarps * 32), smem1,
            stream, p, gpc1); le != cudaSuccess)
        return le;
    if ((err = cudaGetLastError()) != cudaSuccess) return err;
    dim3 g2(max_active, groups2 / gpc2);
    if (const cudaError_t le = launch_k(stream_down_kernel<TA, WQ>, dim3(g2), dim3(kStreamWarps * 32), smem2,
            stream, p, gpc2); le != cudaSuccess)
        return le;
    return cudaGetLastError();
}

// launch_stream_t for one weight format, defined in ffn_stream_<format>.cu so
// that the formats' kernel instantiations compile in parallel
template <int WQ>
cudaError_t launch_stream_w(const FfnProblem& p, cudaStream_t stream);
// int4 weights with fp32 activations (ffn_stream_int4w_f32a.cu)
cudaError_t launch_stream_int4w_f32a(const FfnProblem& p, cudaStream_t stream);

}  // namespace gbmoe
