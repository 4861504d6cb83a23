// Fused MoE with fp8 tensor cores: block-scaled e4m3 weights used as stored.
//
// The route the DeepSeek-V3 recipe implies for its block-FP8 expert weights
// (e4m3, one fp32 scale per 128x128 block, the format of Section 6.2): the
// weight tiles go from HBM to shared memory to tcgen05.mma kind::f8f6f4
// unchanged, with no decode step. The activations entering each GEMM (x,
// then h) are brought to e4m3 per row and 128 consecutive k: with
// s = amax / 448 and v = x / s, a first code q1 = e4m3(v) and a second code
// q2 = e4m3(v - q1) for what the first leaves out, so that x = s * (q1 + q2)
// with an error of at most max(2^-8 |v|, 2^-10) * s (a single e4m3 code would
// leave up to 2^-4 |v|: about 4% of a row's largest output). Each 128-wide k
// block takes two MMA passes, q1 x W and q2 x W, into the same partial sum
// in tensor memory; the epilogue warps promote it,
// acc += P * s * w_scale[n-block][k-block], into fp32 accumulators held in
// registers (the scales change from one k block to the next, so the tensor
// cores cannot accumulate across them).
//
//   quant_rows     x rows in sorted order -> (q1, q2) rows + 1x128 scales
//   gate/up GEMM   -> h = silu(gate) * up (bf16), then h quantised the same way
//   down GEMM      -> y (bf16)
//
// One persistent CTA per SM walks the (M tile, N tile) list built on the
// device. Warp roles (320 threads):
//   warp 0    one lane issues TMA loads of q1 and q2 (128 rows x 128 e4m3
//             each, as two 64-row boxes: the second only when the tile holds
//             rows there) and B (2 x 128 rows x 128 e4m3), 128-byte
//             swizzled, into a 3-stage ring;
//   warp 1    allocates 512 TMEM columns (two 128 x 256 fp32 partial sums)
//             and one lane issues tcgen05.mma (M=128, N=256, K=32): four for
//             q1 and four for q2 per 128-wide k block, alternating between
//             the two partial sums;
//   warps 2-9 promote: warp w reads TMEM lanes 32*(w%4).. (tile rows) and
//             half (w-2)/4 of the columns, accumulates in registers, and at
//             the tile's end applies SwiGLU (gate/up) or stores y.
// For the gate/up GEMM the 256 B rows of a tile are 128 gate rows and the 128
// up rows of the same output columns; a promoting thread holds 64 gate and the
// matching 64 up columns of its row, so SwiGLU needs no exchange.
// Every mbarrier wait is bounded as in the bf16 GEMM (tc_ptx.cuh).
#include <cuda_fp8.h>

#include <cstdlib>

#include "common.cuh"
#include "ffn_sched.h"
#include "kernels.h"
#include "tc_ptx.cuh"

namespace gbmoe {
namespace tcf8 {

using namespace tc;

constexpr int BM = 128, BN = 256, BK = 128;  // BK e4m3 = 128 bytes = one swizzle row
constexpr int QB = 128;                      // quantisation block along k (activations and weights)
constexpr int A_BYTES = BM * BK;             // one activation code plane
constexpr int B_BYTES = BN * BK;
constexpr int STAGES = 3;
constexpr int STAGE_BYTES = 2 * A_BYTES + B_BYTES;  // q1, q2, B
constexpr int PROMOTE_WARPS = 8;
constexpr int THREADS = 64 + PROMOTE_WARPS * 32;
constexpr int TMEM_COLS = 512;  // two 256-column partial sums
constexpr int NUM_BARS = 2 * STAGES + 2 + 2 + 1;
constexpr int SMEM_BYTES = 1024 + STAGES * STAGE_BYTES + NUM_BARS * 8 + 16;
static_assert(SMEM_BYTES <= 232448, "shared memory per CTA");

// Instruction descriptor, kind::f8f6f4: fp32 accumulator (bits 4-5 = 1), A and
// B e4m3 (format 0 in bits 7-9 and 10-12), both K-major, N/8 in bits 17-22,
// M/16 in bits 24-28.
constexpr uint32_t kIdescF8 = (1u << 4) | ((uint32_t)(BN >> 3) << 17) | ((uint32_t)(BM >> 4) << 24);

__device__ __forceinline__ void mma_fp8(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(a_desc), "l"(b_desc), "r"(kIdescF8), "r"(accumulate)
        : "memory");
}

struct Params {
    int K;                  // reduction length (a multiple of 128)
    int n_tiles;            // N tiles per M tile
    int out_cols;           // row length of the output
    int b_rows_per_expert;  // rows of the B tensor per expert
    const int32_t* counts;
    const int32_t* offsets;
    const int32_t* sched;
    int E;
    int64_t n_rows;
    __nv_bfloat16* out;
    int32_t* err;
    const float* a_scale;   // [n_rows, K/128] activation scales
    const float* w_scale0;  // [E, b_rows_per_expert/128, K/128] scales of the B rows in the first /
    const float* w_scale1;  // second half of the tile (gate / up, or down / down)
    uint64_t wait_limit_ns;
};

struct Work {
    int e, m, nt;
    int64_t row0;  // absolute first row of the M tile
    int rows;      // valid rows in the tile
};

__device__ __forceinline__ Work decode_work(const Params& p, int w) {
    const int2* tiles = reinterpret_cast<const int2*>(p.sched + sched_tiles_offset(p.E));
    const int mt = w / p.n_tiles;
    Work r;
    r.nt = w - mt * p.n_tiles;
    const int2 t = tiles[mt];
    r.e = t.x;
    r.m = t.y;
    const int64_t cnt = p.counts ? p.counts[r.e] : p.n_rows;
    r.row0 = (p.offsets ? p.offsets[r.e] : 0) + (int64_t)r.m * BM;
    r.rows = (int)min64(BM, cnt - (int64_t)r.m * BM);
    return r;
}

// first B row (in the stacked [E * rows_per_expert, K] tensor) of each tile half
template <bool SWIGLU>
__device__ __forceinline__ void b_rows(const Params& p, const Work& wk, int& b0, int& b1) {
    b0 = wk.e * p.b_rows_per_expert + (SWIGLU ? wk.nt * (BN / 2) : wk.nt * BN);
    b1 = SWIGLU ? b0 : b0 + BN / 2;
}

// ---------------------------------------------- activation quantisation

// e4m3 codes of (a, b), a in the low byte: round to nearest even, saturating
// at +-448 (the hardware conversion)
__device__ __forceinline__ uint32_t e4m3x2(float a, float b) {
    return (uint32_t)__nv_cvt_float2_to_fp8x2(make_float2(a, b), __NV_SATFINITE, __NV_E4M3);
}

// Rows of a bf16 matrix [*, K] -> two e4m3 code planes q1, q2 [n_rows, K]
// and fp32 scales s [n_rows, K/128]: for every row and 128-wide block,
// amax = max |x|, s = amax / 448 (1 when amax = 0), v = x / s,
// q1 = e4m3(v), q2 = e4m3(v - q1) (v - q1 is exact in fp32); both roundings
// to nearest even, saturating. Row r reads
// source row sorted_pair[r] / pair_div (r itself without sorted_pair; a
// negative entry gives a zero row). One warp per row; lane l takes elements
// 4l .. 4l+3 of every block.
__global__ void __launch_bounds__(256)
quant_rows_kernel(const __nv_bfloat16* __restrict__ src, const int32_t* __restrict__ sorted_pair, int pair_div,
                  int64_t n_rows, int K, uint8_t* __restrict__ q1, uint8_t* __restrict__ q2,
                  float* __restrict__ s) {
    pdl_enter();
    const int lane = threadIdx.x & 31;
    const int64_t warps = (int64_t)gridDim.x * (blockDim.x >> 5);
    const int nblk = K / QB;
    for (int64_t r = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); r < n_rows; r += warps) {
        int64_t srow = r;
        if (sorted_pair) {
            const int32_t pr = sorted_pair[r];
            srow = pr >= 0 ? pr / pair_div : -1;
        }
        constexpr int U = 8;  // blocks whose loads are in flight together
        for (int b0 = 0; b0 < nblk; b0 += U) {
            uint2 raw[U];
#pragma unroll
            for (int u = 0; u < U; ++u) {
                raw[u] = make_uint2(0, 0);
                if (srow >= 0 && b0 + u < nblk)
                    raw[u] = *reinterpret_cast<const uint2*>(src + srow * K + (b0 + u) * QB + 4 * lane);
            }
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int b = b0 + u;
                if (b >= nblk) break;
                const float v[4] = {bf16lo(raw[u].x), bf16hi(raw[u].x), bf16lo(raw[u].y), bf16hi(raw[u].y)};
                float amax = fmaxf(fmaxf(fabsf(v[0]), fabsf(v[1])), fmaxf(fabsf(v[2]), fabsf(v[3])));
#pragma unroll
                for (int d = 16; d >= 1; d >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, d));
                const float sc = amax > 0.0f ? __fdiv_rn(amax, 448.0f) : 1.0f;
                float t[4], rr[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) t[i] = __fdiv_rn(v[i], sc);
                const uint32_t a = e4m3x2(t[0], t[1]) | (e4m3x2(t[2], t[3]) << 16);
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const __half_raw h =
                        __nv_cvt_fp8_to_halfraw((__nv_fp8_storage_t)((a >> (8 * i)) & 0xffu), __NV_E4M3);
                    rr[i] = __fsub_rn(t[i], __half2float(__half(h)));
                }
                const uint32_t a2 = e4m3x2(rr[0], rr[1]) | (e4m3x2(rr[2], rr[3]) << 16);
                *reinterpret_cast<uint32_t*>(q1 + r * K + b * QB + 4 * lane) = a;
                *reinterpret_cast<uint32_t*>(q2 + r * K + b * QB + 4 * lane) = a2;
                if (lane == 0) s[r * nblk + b] = sc;
            }
        }
    }
}

// -------------------------------------------------------------- the GEMM

template <bool SWIGLU>  // gate/up GEMM with the SwiGLU epilogue, or the down GEMM
__global__ void __launch_bounds__(THREADS, 1)
tc_fp8_gemm_kernel(const __grid_constant__ CUtensorMap tm_a1, const __grid_constant__ CUtensorMap tm_a2,
                   const __grid_constant__ CUtensorMap tm_b0, const __grid_constant__ CUtensorMap tm_b1,
                   const Params p) {
    pdl_enter();
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    uint8_t* sA1 = smem;
    uint8_t* sA2 = smem + STAGES * A_BYTES;
    uint8_t* sB = smem + 2 * STAGES * A_BYTES;
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE_BYTES);
    uint64_t* full = bars;                // q1, q2 and B landed
    uint64_t* empty = bars + STAGES;      // MMAs reading the slot finished
    uint64_t* pfull = bars + 2 * STAGES;  // partial sums of one k block ready (2 buffers)
    uint64_t* pempty = pfull + 2;         // partial sums read by every promoting warp
    uint64_t* drain = pfull + 4;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + NUM_BARS);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&pfull[b], 1);
            mbar_init(&pempty[b], PROMOTE_WARPS);
        }
        mbar_init(drain, 1);
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                     "r"(TMEM_COLS)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;

    const int total = p.sched[1] * p.n_tiles;
    const int nkb = p.K / BK;

    if (warp == 0 && lane == 0) {
        // ---------------------------------------------------- TMA producer
        int stage = 0;
        uint32_t phase = 0;
        uint32_t inflight = 0, inflight_par = 0;  // stages loaded but not seen consumed
        bool ok = true;
        for (int w = blockIdx.x; w < total && ok; w += gridDim.x) {
            const Work wk = decode_work(p, w);
            int b0, b1;
            b_rows<SWIGLU>(p, wk, b0, b1);
            // A in two 64-row boxes; the second only when the tile has rows
            // there (the MMA's rows past the tile's end read whatever the slot
            // held, and their accumulators are never stored)
            const bool upper = wk.rows > BM / 2;
            for (int kb = 0; kb < nkb; ++kb) {
                if (!mbar_wait(&empty[stage], phase ^ 1, abort_flag, p.err, p.wait_limit_ns)) { ok = false; break; }
                inflight &= ~(1u << stage);
                mbar_expect_tx(&full[stage], (upper ? 2 * A_BYTES : A_BYTES) + B_BYTES);
                tma_load_2d(sA1 + stage * A_BYTES, &tm_a1, kb * BK, (int)wk.row0, &full[stage]);
                tma_load_2d(sA2 + stage * A_BYTES, &tm_a2, kb * BK, (int)wk.row0, &full[stage]);
                if (upper) {
                    tma_load_2d(sA1 + stage * A_BYTES + A_BYTES / 2, &tm_a1, kb * BK, (int)wk.row0 + BM / 2, &full[stage]);
                    tma_load_2d(sA2 + stage * A_BYTES + A_BYTES / 2, &tm_a2, kb * BK, (int)wk.row0 + BM / 2, &full[stage]);
                }
                tma_load_2d(sB + stage * B_BYTES, &tm_b0, kb * BK, b0, &full[stage]);
                tma_load_2d(sB + stage * B_BYTES + B_BYTES / 2, &tm_b1, kb * BK, b1, &full[stage]);
                inflight |= 1u << stage;
                inflight_par = (inflight_par & ~(1u << stage)) | (phase << stage);
                if (++stage == STAGES) { stage = 0; phase ^= 1; }
            }
        }
        for (int s = 0; s < STAGES; ++s)
            if ((inflight >> s) & 1u) drain_wait(&full[s], (inflight_par >> s) & 1u);
    } else if (warp == 1 && lane == 0) {
        // ------------------------------------------------------ MMA issuer
        int stage = 0;
        uint32_t phase = 0;
        uint32_t kbg = 0;  // k blocks issued so far: partial buffer kbg & 1, its use (kbg >> 1)
        bool ok = true;
        bool issued = false;
        for (int w = blockIdx.x; w < total && ok; w += gridDim.x) {
            for (int kb = 0; kb < nkb; ++kb, ++kbg) {
                const uint32_t pb = kbg & 1u, pph = (kbg >> 1) & 1u;
                if (!mbar_wait(&pempty[pb], pph ^ 1, abort_flag, p.err, p.wait_limit_ns)) { ok = false; break; }
                if (!mbar_wait(&full[stage], phase, abort_flag, p.err, p.wait_limit_ns)) { ok = false; break; }
                tc_fence_after();
                const uint64_t da1 = sw128_desc(smem_u32(sA1 + stage * A_BYTES));
                const uint64_t da2 = sw128_desc(smem_u32(sA2 + stage * A_BYTES));
                const uint64_t db = sw128_desc(smem_u32(sB + stage * B_BYTES));
                const uint32_t d_tmem = tmem_base + pb * BN;
#pragma unroll
                for (int j = 0; j < BK / 32; ++j)  // +32 bytes along K per instruction
                    mma_fp8(d_tmem, da1 + 2 * j, db + 2 * j, j != 0 ? 1u : 0u);
#pragma unroll
                for (int j = 0; j < BK / 32; ++j)  // the residual codes into the same partial sum
                    mma_fp8(d_tmem, da2 + 2 * j, db + 2 * j, 1u);
                issued = true;
                mma_commit(&empty[stage]);
                mma_commit(&pfull[pb]);
                if (++stage == STAGES) { stage = 0; phase ^= 1; }
            }
        }
        if (issued) {  // every MMA issued has finished before TMEM is released
            mma_commit(drain);
            drain_wait(drain, 0);
        }
    } else if (warp >= 2) {
        // ------------------------------------------ promotion and epilogue
        const int q = warp & 3;            // TMEM lane quarter of this warp
        const int half = (warp - 2) >> 2;  // which half of the tile's columns
        const int r = q * 32 + lane;       // tile row of this thread
        const uint32_t t_row = tmem_base + ((uint32_t)(q * 32) << 16);
        const int kq = p.K / QB;
        const int nb_per_e = p.b_rows_per_expert / QB;
        // this thread's 128 columns: 64 gate + the matching 64 up (SwiGLU), or 128 down
        const int c0 = SWIGLU ? 64 * half : 128 * half;
        const int c1 = SWIGLU ? BN / 2 + 64 * half : 128 * half + 64;
        uint32_t kbg = 0;
        for (int w = blockIdx.x; w < total; w += gridDim.x) {
            // scales: the activation row's, and the weight n-blocks of this
            // thread's columns, as element offsets (int: the library refuses
            // fp8 configs whose scale tensors reach 2^31 entries)
            int sa_off, s_off;
            {
                const Work wk = decode_work(p, w);
                const int64_t row = wk.row0 + r;
                sa_off = row < p.n_rows ? (int)(row * kq) : -1;
                // gate/up: 128 gate rows nt*128.. are n-block nt of the gate scales, up the same;
                // down: columns 128*half .. are n-block 2*nt + half
                s_off = (wk.e * nb_per_e + (SWIGLU ? wk.nt : 2 * wk.nt + half)) * kq;
            }
            float acc[128];
#pragma unroll
            for (int i = 0; i < 128; ++i) acc[i] = 0.0f;
            // the k block's scales, loaded one k block ahead (a k block of
            // MMAs takes far longer than a load) so that the promotion does
            // not wait on them
            auto scales_of = [&](int kb, float& a, float& w0, float& w1) {
                const bool ok_kb = kb < nkb;
                a = sa_off >= 0 && ok_kb ? p.a_scale[sa_off + kb] : 0.0f;
                w0 = ok_kb ? p.w_scale0[s_off + kb] : 0.0f;
                w1 = ok_kb ? p.w_scale1[s_off + kb] : 0.0f;  // the same block of the up (or down) scales
            };
            float a0, x0, y0;
            scales_of(0, a0, x0, y0);
            bool ok = true;
            for (int kb = 0; kb < nkb; ++kb, ++kbg) {
                const uint32_t pb = kbg & 1u, pph = (kbg >> 1) & 1u;
                const float f0 = a0 * x0, f1 = a0 * y0;
                scales_of(kb + 1, a0, x0, y0);
                if (!warp_wait(&pfull[pb], pph, abort_flag, p.err, p.wait_limit_ns)) { ok = false; break; }
                tc_fence_after();
                const uint32_t tb = t_row + pb * BN;
                // 16 columns at a time: next to 128 accumulators, wider loads spill
#pragma unroll
                for (int part = 0; part < 8; ++part) {
                    float v[16];
                    tmem_ld16(tb + (uint32_t)((part < 4 ? c0 : c1) + 16 * (part & 3)), v);
                    const float f = part < 4 ? f0 : f1;
#pragma unroll
                    for (int i = 0; i < 16; ++i) acc[16 * part + i] = fmaf(v[i], f, acc[16 * part + i]);
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&pempty[pb]);
            }
            if (!ok) break;
            const Work wk = decode_work(p, w);
            const int64_t row = wk.row0 + r;
            if (r < wk.rows) {
                if constexpr (SWIGLU) {
                    __nv_bfloat16* dst = p.out + row * (int64_t)p.out_cols + wk.nt * (BN / 2) + 64 * half;
#pragma unroll
                    for (int c = 0; c < 8; ++c) {
                        float h[8];
#pragma unroll
                        for (int i = 0; i < 8; ++i) h[i] = silu_mul(acc[8 * c + i], acc[64 + 8 * c + i]);
                        uint4 u;
                        u.x = pack_bf16x2(h[0], h[1]);
                        u.y = pack_bf16x2(h[2], h[3]);
                        u.z = pack_bf16x2(h[4], h[5]);
                        u.w = pack_bf16x2(h[6], h[7]);
                        reinterpret_cast<uint4*>(dst)[c] = u;
                    }
                } else {
                    __nv_bfloat16* dst = p.out + row * (int64_t)p.out_cols + wk.nt * BN + 128 * half;
#pragma unroll
                    for (int c = 0; c < 16; ++c) {
                        uint4 u;
                        u.x = pack_bf16x2(acc[8 * c + 0], acc[8 * c + 1]);
                        u.y = pack_bf16x2(acc[8 * c + 2], acc[8 * c + 3]);
                        u.z = pack_bf16x2(acc[8 * c + 4], acc[8 * c + 5]);
                        u.w = pack_bf16x2(acc[8 * c + 6], acc[8 * c + 7]);
                        reinterpret_cast<uint4*>(dst)[c] = u;
                    }
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(TMEM_COLS)
                     : "memory");
    }
}

// ------------------------------------------------------------------- host

// e4m3 matrix [rows, K] in {128 bytes, box_rows rows} boxes, 128-byte swizzle
static bool map_e4m3(CUtensorMap* m, const void* base, int64_t rows, int64_t K, int box_rows) {
    return make_map(m, base, rows, K, CU_TENSOR_MAP_DATA_TYPE_UINT8, 1, BK, CU_TENSOR_MAP_SWIZZLE_128B, box_rows);
}

// q holds the two code planes [2, n_rows, K]
static cudaError_t launch_quant(const void* src, const int32_t* sorted_pair, int pair_div, int64_t n_rows, int K,
                                void* q, float* s, cudaStream_t stream) {
    const int blocks = (int)min64((n_rows + 7) / 8, (int64_t)sm_count() * 16);
    if (blocks <= 0) return cudaSuccess;
    if (const cudaError_t le = launch_k(quant_rows_kernel, dim3(blocks), dim3(256), 0, stream,
            static_cast<const __nv_bfloat16*>(src), sorted_pair, pair_div, n_rows, K, static_cast<uint8_t*>(q),
            static_cast<uint8_t*>(q) + n_rows * K, s);
        le != cudaSuccess)
        return le;
    return cudaGetLastError();
}

template <bool SWIGLU>
static cudaError_t launch_gemm(const CUtensorMap& a1, const CUtensorMap& a2, const CUtensorMap& b0,
                               const CUtensorMap& b1, const Params& prm, int64_t max_work, cudaStream_t stream) {
    static DeviceOnce smem_set;
    cudaError_t e = smem_set.run([] {
        return cudaFuncSetAttribute(tc_fp8_gemm_kernel<SWIGLU>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    SMEM_BYTES);
    });
    if (e != cudaSuccess) return e;
    const int grid = (int)min64(sm_count(), max_work);
    if (grid <= 0) return cudaSuccess;
    if (const cudaError_t le = launch_k(tc_fp8_gemm_kernel<SWIGLU>, dim3(grid), dim3(THREADS), SMEM_BYTES, stream, a1, a2,
                                        b0, b1, prm);
        le != cudaSuccess)
        return le;
    return cudaGetLastError();
}

}  // namespace tcf8

bool ffn_tc_fp8_supported(const FfnProblem& p) {
    return p.act_dtype == GBMOE_BF16 && p.w_dtype == GBMOE_FP8_E4M3_B128 && p.H % 256 == 0 && p.I % 128 == 0 &&
           tc::encode_fn() != nullptr;
}

cudaError_t launch_ffn_tc_fp8(const FfnProblem& p, cudaStream_t stream) {
    using namespace tcf8;
    if (p.n_rows == 0) return cudaSuccess;
    cudaError_t err = launch_ffn_schedule(p.counts, p.E, p.n_rows, BM, p.sched, stream);
    if (err != cudaSuccess) return err;
    // x rows in sorted order (x itself for the shared expert), quantised per 1x128
    if ((err = launch_quant(p.x, p.sorted_pair, p.pair_div, p.n_rows, p.H, p.a_q, p.a_s, stream)) != cudaSuccess)
        return err;
    const int64_t max_m = sched_max_tiles(p.E, p.n_rows, BM);
    const uint8_t* aq = static_cast<const uint8_t*>(p.a_q);
    const uint8_t* hq = static_cast<const uint8_t*>(p.h_q);
    CUtensorMap ma1, ma2, mg, mu, mh1, mh2, md;
    if (!map_e4m3(&ma1, aq, p.n_rows, p.H, BM / 2) || !map_e4m3(&ma2, aq + p.n_rows * p.H, p.n_rows, p.H, BM / 2) ||
        !map_e4m3(&mg, p.w_gate, (int64_t)p.E * p.I, p.H, BN / 2) ||
        !map_e4m3(&mu, p.w_up, (int64_t)p.E * p.I, p.H, BN / 2) || !map_e4m3(&mh1, hq, p.n_rows, p.I, BM / 2) ||
        !map_e4m3(&mh2, hq + p.n_rows * p.I, p.n_rows, p.I, BM / 2) ||
        !map_e4m3(&md, p.w_down, (int64_t)p.E * p.H, p.I, BN / 2))
        return cudaErrorInvalidValue;
    Params g{};
    g.K = p.H; g.n_tiles = p.I / (BN / 2); g.out_cols = p.I; g.b_rows_per_expert = p.I;
    g.counts = p.counts; g.offsets = p.offsets; g.sched = p.sched; g.E = p.E; g.n_rows = p.n_rows;
    g.out = static_cast<__nv_bfloat16*>(p.h); g.err = p.err;
    g.a_scale = p.a_s;
    g.w_scale0 = static_cast<const float*>(p.s_gate); g.w_scale1 = static_cast<const float*>(p.s_up);
    g.wait_limit_ns = tc_wait_limit_ns();
    if ((err = launch_gemm<true>(ma1, ma2, mg, mu, g, max_m * g.n_tiles, stream)) != cudaSuccess) return err;
    // h quantised per 1x128 for the down GEMM
    if ((err = launch_quant(p.h, nullptr, 1, p.n_rows, p.I, p.h_q, p.h_s, stream)) != cudaSuccess) return err;
    Params d = g;
    d.K = p.I; d.n_tiles = p.H / BN; d.out_cols = p.H; d.b_rows_per_expert = p.H;
    d.out = static_cast<__nv_bfloat16*>(p.y);
    d.a_scale = p.h_s;
    d.w_scale0 = static_cast<const float*>(p.s_down); d.w_scale1 = d.w_scale0;
    return launch_gemm<false>(mh1, mh2, md, md, d, max_m * d.n_tiles, stream);
}

}  // namespace gbmoe
