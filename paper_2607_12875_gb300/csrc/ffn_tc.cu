// Fused MoE on tensor cores: grouped GEMMs with tcgen05, TMEM and TMA.
//
// Rows of each expert are contiguous after the permutation, so every M tile
// is a block of consecutive sorted rows of one expert. A tile that runs past
// its expert's last row computes rows of the next expert (or zero fill past
// the end); those rows are never stored.
//
// One persistent CTA per SM (CG = 1) or per pair of SMs (CG = 2) walks the
// (M tile, N tile) list built on the device. Warp roles:
//   warp 0    one lane issues TMA loads into a ring of stages: the A tile
//             (128 x 64 bf16, 128-byte swizzled) and the B tile (two 128-row
//             halves: 128 gate + 128 up rows, or 256 down rows), or the raw
//             quantised B tile instead of B;
//   warp 1    allocates 512 TMEM columns (two 128 x 256 fp32 accumulators)
//             and one lane issues tcgen05.mma (kind::f16, M=128 or 256 for a
//             pair, N=256, K=16), releasing ring slots and accumulators
//             through tcgen05.commit -> mbarrier;
//   warps 2-5 read the accumulator with tcgen05.ld (warp w owns TMEM lanes
//             32*(w%4)..+31, i.e. tile rows) and produce the results: h =
//             silu(gate) * up for the gate/up GEMM, y for the down GEMM
//             (TMA stores through a swizzled staging buffer), fp32 logits for
//             the router, or the fused Weight Sum's weighted slots;
//   warps 6+  quantised weights (fp8 e4m3 with 128x128 block scales, int4
//             with 128-wide group scales, MXFP4 with 32-wide E8M0 scales):
//             one thread per B row decodes the raw tile, applies the scale
//             and writes the bf16 operand in the swizzled layout the MMA
//             reads; bf16 weights on one CTA: four warps gather the A rows of
//             the gate/up GEMM from x (cp.async), so no sorted copy of x is
//             written.
// A CTA pair (tcgen05 cta_group::2) shares each MMA: each CTA holds 128 A
// rows and half of the B rows; the odd CTA's loads complete on the even
// CTA's barriers and the even CTA's commits arrive on both CTAs' barriers.
// When experts have many rows, so that several M tiles would decode the same
// weight tile again, the caller's workspace instead receives one bf16 copy
// of the active experts' weights (dequant_weights_kernel, same decode) and
// the bf16 GEMM runs on it.
// Every mbarrier wait is bounded (two seconds by default); on expiry the CTA
// sets the device error word, stops issuing work, drains what it issued and
// frees its TMEM.
#include <cuda.h>
#include <cuda_fp16.h>


#include "common.cuh"
#include "ffn_sched.h"
#include "kernels.h"
#include "tc_ptx.cuh"

namespace gbmoe {
namespace tc {

constexpr int BM = 128, BN = 256, BK = 64;  // BK bf16 = 128 bytes = one swizzle row
constexpr int A_BYTES = BM * BK * 2;
constexpr int B_BYTES = BN * BK * 2;  // bf16 B tile of one MMA (a CTA of a pair holds half)
constexpr int TMEM_COLS = 512;
constexpr int kFp8PrefetchAhead = 4;  // k-blocks the fp8 producer prefetches into L2 ahead of its loads

// Bytes of the raw weight tile (BN rows x BK elements) TMA brings in; 0: B is
// loaded as bf16 directly.
template <int WQ>
struct Fmt;
template <>
struct Fmt<GBMOE_BF16> {
    static constexpr int RAW_BYTES = 0;
};
template <>
struct Fmt<GBMOE_FP8_E4M3_B128> {
    static constexpr int RAW_BYTES = BN * BK;
};
template <>
struct Fmt<GBMOE_INT4_G128> {
    static constexpr int RAW_BYTES = BN * BK / 2;
};
template <>
struct Fmt<GBMOE_MXFP4> {
    static constexpr int RAW_BYTES = BN * BK / 2;
};

// nibble-packed formats: a raw row of BK elements is BK / 2 bytes
template <int WQ>
constexpr bool packed4() { return WQ == GBMOE_INT4_G128 || WQ == GBMOE_MXFP4; }

// Per weight format WQ and CTA group CG: CG = 1, one CTA per 128 x 256 tile;
// CG = 2, a CTA pair per 256 x 256 tile, each CTA holding 128 A rows and 128
// of the 256 B rows (bf16 B only: quantised weights are decoded beforehand
// for pairs). Pipeline depth as shared memory allows.
template <int WQ, int CG>
struct Cfg {
    static_assert(CG == 1 || WQ == GBMOE_BF16, "CTA pairs take bf16 B tiles");
    static constexpr int RAW = Fmt<WQ>::RAW_BYTES / CG;  // raw B bytes per stage of one CTA
    static constexpr int B_HELD = B_BYTES / CG;          // bf16 B bytes per stage of one CTA
    static constexpr int B_ROWS = BN / CG;               // B rows of one CTA
    static constexpr int CONVERT_WARPS = RAW ? B_ROWS / 32 : 0;  // one thread per B row
    // bf16, one CTA: four warps can gather the A rows from x themselves (one
    // thread per row; 10 warps keep a thread's 168 registers)
    static constexpr bool GATHER = WQ == GBMOE_BF16 && CG == 1;
    static constexpr int GATHER_WARPS = GATHER ? BM / 32 : 0;
    static constexpr int GATHER_AHEAD = 2;  // k blocks a gather warp keeps in flight before signalling
    static constexpr int THREADS = 192 + CONVERT_WARPS * 32 + GATHER_WARPS * 32;
    static constexpr int STAGES = CG == 1 ? (WQ == GBMOE_FP8_E4M3_B128 ? 3 : 4) : (RAW ? 5 : 6);
};

template <int WQ, int CG>
struct Layout {
    using C = Cfg<WQ, CG>;
    static constexpr int STAGES = C::STAGES;
    static constexpr int STAGE_BYTES = A_BYTES + C::B_HELD + C::RAW;
    static constexpr int NUM_BARS = 3 * STAGES + 4 + 1;
    static constexpr int BASE_BYTES = 1024 + STAGES * STAGE_BYTES + NUM_BARS * 8 + 16;
    // output staging for TMA stores: 4 epilogue warps x 2 buffers x (32 rows x 64 bytes),
    // when it fits next to the ring (otherwise the epilogue stores from registers)
    static constexpr int EPI_BYTES = BASE_BYTES + 4 * 2 * 2048 <= 232448 ? 4 * 2 * 2048 : 0;
    static constexpr int SMEM_BYTES = BASE_BYTES + EPI_BYTES;
    static_assert(SMEM_BYTES <= 232448, "shared memory per CTA");
};

struct Params {
    int K;                 // reduction length
    int n_tiles;           // N tiles per M tile
    int out_cols;          // row length of the output
    int b_rows_per_expert; // rows of the B tensor per expert
    int swiglu;            // 1: gate/up GEMM with SwiGLU epilogue; 0: plain output
    const int32_t* counts;
    const int32_t* offsets;
    const int32_t* sched;
    int E;
    int64_t n_rows;
    __nv_bfloat16* out;
    int32_t* err;
    const void* scale0;  // scales of the B rows in the first / second half of the tile
    const void* scale1;
    uint64_t wait_limit_ns;  // limit of each pipeline wait (kWaitLimitNs unless a test shortens it)
    // fp32 output instead of bf16 (the router's logits): out_f32[row, col] =
    // accumulator (+ col_bias[col]) for col < f32_cols; out is unused then
    float* out_f32;
    const float* col_bias;
    int f32_cols;
    // Weight Sum fused into the down GEMM (fuse_k > 0, the layer's top_k): row
    // r is pair p = sorted_pair[r] = t*k + j; its output times topk_w[p] goes to
    // slots[p] (pair order, bf16), and the thread completing the k-th arrival of
    // token t on this N tile (arrive[t * n_tiles + nt]) sums the token's k
    // slots in order j = 0..k-1, adds y_shared[t] and writes out_final[t].
    int fuse_k;
    const int32_t* sorted_pair;
    const float* topk_w;
    const __nv_bfloat16* y_shared;
    __nv_bfloat16* out_final;
    int32_t* arrive;
    // A rows gathered from x by the kernel (Cfg::GATHER; null: A by TMA):
    // row r of the sorted order is x row a_gather[r] / a_gather_div (a
    // negative entry, and rows past n_rows, read x row 0; never stored)
    const int32_t* a_gather;
    int a_gather_div;
    const __nv_bfloat16* a_src;  // x [*, K]
};

// 16-byte global -> shared copy through L2 (cp.async), tracked by commit groups
__device__ __forceinline__ void cp_async_16(void* dst, const void* src) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(dst)), "l"(src) : "memory");
}

// Instruction descriptor, kind::f16: fp32 accumulator (bits 4-5 = 1), bf16 A
// and B (bits 7-9, 10-12 = 1), both K-major, N/8 in bits 17-22, M/16 in 24-28
// (M = 128 per CTA, 256 for a CTA pair).
template <int CG>
constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(BN >> 3) << 17) |
                            ((uint32_t)((BM * CG) >> 4) << 24);

template <int CG>
__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t accumulate) {
    if constexpr (CG == 1)
        asm volatile(
            "{\n\t.reg .pred p;\n\t"
            "setp.ne.b32 p, %4, 0;\n\t"
            "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
            "l"(a_desc), "l"(b_desc), "r"(kIdesc<1>), "r"(accumulate)
            : "memory");
    else
        asm volatile(
            "{\n\t.reg .pred p;\n\t"
            "setp.ne.b32 p, %4, 0;\n\t"
            "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
            "l"(a_desc), "l"(b_desc), "r"(kIdesc<2>), "r"(accumulate)
            : "memory");
}

// completion of the MMAs issued so far -> one arrival on `bar` (CG = 2: on
// the barrier at the same offset in each CTA of cta_mask)
template <int CG>
__device__ __forceinline__ void commit_to(uint64_t* bar, uint16_t cta_mask) {
    if constexpr (CG == 1) mma_commit(bar);
    else mma_commit_pair(bar, cta_mask);
}

template <int CG>
__device__ __forceinline__ void tmem_alloc(uint32_t* slot) {
    if constexpr (CG == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(slot)),
                     "r"(TMEM_COLS)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    } else {
        asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(slot)),
                     "r"(TMEM_COLS)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
    }
}

template <int CG>
__device__ __forceinline__ void tmem_dealloc(uint32_t base) {
    if constexpr (CG == 1)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(base), "r"(TMEM_COLS) : "memory");
    else
        asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(base), "r"(TMEM_COLS) : "memory");
}

// 32 fp32 -> 32 bf16 into row `lane` of a 32-row x 64-byte staging buffer in
// the 64-byte-swizzled layout TMA reads for a {32 columns, 32 rows} box
__device__ __forceinline__ void stage_bf16x32(uint8_t* buf, int lane, const float (&v)[32]) {
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        uint4 u;
        u.x = pack_bf16x2(v[8 * q + 0], v[8 * q + 1]);
        u.y = pack_bf16x2(v[8 * q + 2], v[8 * q + 3]);
        u.z = pack_bf16x2(v[8 * q + 4], v[8 * q + 5]);
        u.w = pack_bf16x2(v[8 * q + 6], v[8 * q + 7]);
        *reinterpret_cast<uint4*>(buf + lane * 64 + ((q ^ ((lane >> 1) & 3)) << 4)) = u;
    }
}

__device__ __forceinline__ void store_bf16x32(__nv_bfloat16* dst, const float (&v)[32]) {
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        uint4 u;
        u.x = pack_bf16x2(v[8 * q + 0], v[8 * q + 1]);
        u.y = pack_bf16x2(v[8 * q + 2], v[8 * q + 3]);
        u.z = pack_bf16x2(v[8 * q + 4], v[8 * q + 5]);
        u.w = pack_bf16x2(v[8 * q + 6], v[8 * q + 7]);
        reinterpret_cast<uint4*>(dst)[q] = u;
    }
}

// ----------------------------------------------------- weight decoding

// same for rows of 64 bytes (chunks 0..3) and 32 bytes (chunks 0..1) as TMA
// writes them with 64- and 32-byte swizzling
__device__ __forceinline__ uint32_t sw64_off(int r, int c) { return (uint32_t)(r * 64 + ((c ^ ((r >> 1) & 3)) << 4)); }
__device__ __forceinline__ uint32_t sw32_off(int r, int c) { return (uint32_t)(r * 32 + ((c ^ ((r >> 2) & 1)) << 4)); }

// 16 e4m3 weights (one 16-byte raw chunk) times the block scale -> 16 bf16 in two 16-byte chunks
__device__ __forceinline__ void decode_fp8_16(const uint4 raw, float sc, uint4& o0, uint4& o1) {
    const uint32_t w[4] = {raw.x, raw.y, raw.z, raw.w};
    uint32_t packed[8];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        float2 a = e4m3x2_to_f32x2(w[i] & 0xffffu);
        float2 b = e4m3x2_to_f32x2(w[i] >> 16);
        packed[2 * i] = pack_bf16x2(a.x * sc, a.y * sc);
        packed[2 * i + 1] = pack_bf16x2(b.x * sc, b.y * sc);
    }
    o0 = make_uint4(packed[0], packed[1], packed[2], packed[3]);
    o1 = make_uint4(packed[4], packed[5], packed[6], packed[7]);
}

// 8 int4 weights (one 32-bit word, element 0 in the low nibble) times the
// group scale -> 8 bf16 (one 16-byte chunk). A nibble v becomes the bf16
// 128 + (v xor 8) by OR-ing it into the mantissa of 128.0, and 136 is
// subtracted exactly, which leaves the two's-complement value; then one bf16
// multiply by the scale.
__device__ __forceinline__ uint4 decode_int4_8(uint32_t w, __nv_bfloat162 sc2) {
    const __nv_bfloat162 k136 = __floats2bfloat162_rn(136.0f, 136.0f);
    uint32_t p[4];  // p[i] holds elements (i, i + 4)
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        uint32_t t = ((w >> (4 * i)) & 0x000f000fu) ^ 0x43084308u;
        __nv_bfloat162 v = *reinterpret_cast<__nv_bfloat162*>(&t);
        v = __hmul2(__hsub2(v, k136), sc2);
        p[i] = *reinterpret_cast<uint32_t*>(&v);
    }
    return make_uint4(__byte_perm(p[0], p[1], 0x5410), __byte_perm(p[2], p[3], 0x5410),
                      __byte_perm(p[0], p[1], 0x7632), __byte_perm(p[2], p[3], 0x7632));
}

// 8 FP4 E2M1 weights (one 32-bit word, element 0 in the low nibble) times the
// E8M0 block scale (sc2 = 2^(s-127) in both halves) -> 8 bf16 (one 16-byte
// chunk), exact. A code's exponent and mantissa bits are placed in the bf16
// exponent field 0..3 and top mantissa bit, which reads as the value times
// 2^-126 (the E2M1 subnormal 0.5 as the bf16 subnormal 2^-127); one bf16
// multiply by 2^126 and one by the scale, both exact.
__device__ __forceinline__ uint4 decode_mxfp4_8(uint32_t w, __nv_bfloat162 sc2) {
    const uint32_t k2p126 = 0x7e807e80u;  // bf16x2 (2^126, 2^126)
    uint32_t p[4];  // p[i] holds elements (i, i + 4)
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const uint32_t t = (w >> (4 * i)) & 0x000f000fu;
        uint32_t b = ((t & 0x00080008u) << 12) | ((t & 0x00070007u) << 6);
        __nv_bfloat162 v = __hmul2(*reinterpret_cast<__nv_bfloat162*>(&b),
                                   *reinterpret_cast<const __nv_bfloat162*>(&k2p126));
        v = __hmul2(v, sc2);
        p[i] = *reinterpret_cast<uint32_t*>(&v);
    }
    return make_uint4(__byte_perm(p[0], p[1], 0x5410), __byte_perm(p[2], p[3], 0x5410),
                      __byte_perm(p[0], p[1], 0x7632), __byte_perm(p[2], p[3], 0x7632));
}

// E8M0 byte -> bf16x2 (2^(s-127), 2^(s-127)); s = 0 is the bf16 subnormal 2^-127
__device__ __forceinline__ __nv_bfloat162 e8m0_bf16x2(uint32_t s) {
    const uint32_t h = s ? (s << 7) : 0x0040u;
    const uint32_t b = h | (h << 16);
    return *reinterpret_cast<const __nv_bfloat162*>(&b);
}

// ------------------------------------------------------------------ kernel

struct Work {
    int e, m, nt;
    int64_t row0;  // absolute first row of this CTA's 128 rows of the M tile
    int rows;      // valid rows among them (<= 0: none)
};

// Work item w: M tile w / n_tiles of the list (BM * CG rows of one expert),
// N tile w % n_tiles; CTA `rank` of a pair takes the tile's rows rank*BM ..
template <int CG>
__device__ __forceinline__ Work decode_work(const Params& p, int w, uint32_t rank) {
    const int2* tiles = reinterpret_cast<const int2*>(p.sched + sched_tiles_offset(p.E));
    const int mt = w / p.n_tiles;
    Work r;
    r.nt = w - mt * p.n_tiles;
    const int2 t = tiles[mt];
    r.e = t.x;
    r.m = t.y;
    const int64_t cnt = p.counts ? p.counts[r.e] : p.n_rows;
    const int64_t first = (int64_t)r.m * (BM * CG) + (int64_t)rank * BM;
    r.row0 = (p.offsets ? p.offsets[r.e] : 0) + first;
    r.rows = (int)min64(BM, cnt - first);
    return r;
}

// first B row (in the stacked [E * rows_per_expert, K] tensor) of each tile half
__device__ __forceinline__ void b_rows(const Params& p, const Work& wk, int& b0, int& b1) {
    b0 = wk.e * p.b_rows_per_expert + (p.swiglu ? wk.nt * (BN / 2) : wk.nt * BN);
    b1 = p.swiglu ? b0 : b0 + BN / 2;
}

// Weight Sum of the fused down GEMM, called by a whole epilogue warp after
// its lanes stored their weighted slot rows (columns col0 .. col0 + BN of pair
// `pair`, for the lanes with `valid`). Each such lane counts the arrival of
// its token on this column range; the tokens whose k-th arrival this was are
// then reduced by the whole warp, lane l taking 8 columns: the token's slots
// in slot order (fp32, the same sum whichever warp does it), plus the shared
// expert's row, rounded once; the counter is reset for the next call.
__device__ __noinline__ void fused_weight_sum(const Params& p, bool valid, int64_t pair, int col0) {
    const int lane = threadIdx.x & 31;
    const int k = p.fuse_k;
    const int64_t t = pair / k;
    int32_t* cnt = p.arrive + t * p.n_tiles + col0 / BN;
    bool last = false;
    if (valid) {
        __threadfence();  // the slot row is visible before the arrival is
        last = atomicAdd(cnt, 1) == k - 1;
    }
    uint32_t done = __ballot_sync(0xffffffffu, last);
    if (!done) return;
    __threadfence();  // every slot row of those tokens is visible now
    const int64_t H = p.out_cols;
    while (done) {
        const int src = __ffs(done) - 1;
        done &= done - 1;
        const int64_t tt = __shfl_sync(0xffffffffu, t, src);
        if (lane == src) *cnt = 0;  // ready for the next call
        for (int c = 8 * lane; c < BN; c += 256) {
            float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
            for (int j = 0; j < k; ++j) {
                // other SMs wrote these rows during this kernel: read them from L2
                const uint4 u = __ldcg(reinterpret_cast<const uint4*>(p.out + (tt * k + j) * H + col0 + c));
                const float v[8] = {bf16lo(u.x), bf16hi(u.x), bf16lo(u.y), bf16hi(u.y),
                                    bf16lo(u.z), bf16hi(u.z), bf16lo(u.w), bf16hi(u.w)};
#pragma unroll
                for (int i = 0; i < 8; ++i) acc[i] = __fadd_rn(acc[i], v[i]);
            }
            if (p.y_shared) {
                float v[8];
                Vec8<__nv_bfloat16>::load(p.y_shared + tt * H + col0 + c, v);
#pragma unroll
                for (int i = 0; i < 8; ++i) acc[i] = __fadd_rn(acc[i], v[i]);
            }
            Vec8<__nv_bfloat16>::store(p.out_final + tt * H + col0 + c, acc);
        }
    }
}

template <int WQ, int CG>
__global__ void __launch_bounds__(Cfg<WQ, CG>::THREADS, 1)
tc_gemm_kernel(const __grid_constant__ CUtensorMap tm_a, const __grid_constant__ CUtensorMap tm_b0,
               const __grid_constant__ CUtensorMap tm_b1, const __grid_constant__ CUtensorMap tm_out, const Params p) {
    pdl_enter();
    using C = Cfg<WQ, CG>;
    using L = Layout<WQ, CG>;
    constexpr int STAGES = L::STAGES;
    constexpr int RAW = C::RAW;
    constexpr int BH = C::B_HELD;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    uint8_t* sA = smem;
    uint8_t* sB = smem + STAGES * A_BYTES;
    uint8_t* sR = smem + STAGES * (A_BYTES + BH);  // raw quantised B tiles
    uint8_t* sE = smem + STAGES * L::STAGE_BYTES;  // output staging (L::EPI_BYTES)
    uint64_t* bars = reinterpret_cast<uint64_t*>(sE + L::EPI_BYTES);
    uint64_t* full = bars;                 // TMA landed (A + B or A + raw B)
    uint64_t* empty = bars + STAGES;       // MMAs reading the slot finished
    uint64_t* conv = bars + 2 * STAGES;    // bf16 B written by the converters
    uint64_t* tfull = bars + 3 * STAGES;
    uint64_t* tempty = bars + 3 * STAGES + 2;
    uint64_t* drain = bars + 3 * STAGES + 4;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + L::NUM_BARS);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t rank = CG == 2 ? cluster_rank() : 0u;  // 0: this CTA issues the MMAs
    if (threadIdx.x == 0) {
        const bool gathering = C::GATHER && p.a_gather != nullptr;
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&full[s], gathering ? 1 + C::GATHER_WARPS : 1);  // + one arrival per gather warp
            mbar_init(&empty[s], 1);
            mbar_init(&conv[s], C::CONVERT_WARPS ? C::CONVERT_WARPS : 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(&tfull[a], 1);
            mbar_init(&tempty[a], 4 * CG);  // one arrival per epilogue warp of each CTA
        }
        mbar_init(drain, 1);
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 1) tmem_alloc<CG>(tmem_slot);
    tc_fence_before();
    __syncthreads();
    if constexpr (CG == 2) cluster_sync();  // both CTAs' barriers exist before either signals the other
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;

    const int total = p.sched[1] * p.n_tiles;
    const int nkb = p.K / BK;
    const int unit = blockIdx.x / CG, n_units = gridDim.x / CG;  // CTA pairs walk the list together

    if (warp == 0 && lane == 0) {
        // ---------------------------------------------------- TMA producer
        // CG = 2: both CTAs' copies of a slot complete on the even CTA's
        // full barrier, which expects the bytes of both
        int stage = 0;
        uint32_t phase = 0;
        uint32_t inflight = 0, inflight_par = 0;  // stages loaded but not seen consumed
        bool ok = true;
        for (int w = unit; w < total && ok; w += n_units) {
            const Work wk = decode_work<CG>(p, w, rank);
            int b0, b1;
            b_rows(p, wk, b0, b1);
            // CG = 2: this CTA's half of the B tile (gate rows / up rows, or down rows 0-127 / 128-255)
            const CUtensorMap* tm_bh = rank ? &tm_b1 : &tm_b0;
            const int bh = rank ? b1 : b0;
            for (int kb = 0; kb < nkb; ++kb) {
                if (WQ == GBMOE_FP8_E4M3_B128 && kb + kFp8PrefetchAhead < nkb) {
                    // fp8 tiles wait on the decode as well as on the load: bring the
                    // k-block a few stages ahead into L2 so its TMA load returns sooner
                    const int xp = (kb + kFp8PrefetchAhead) * BK;
                    tma_prefetch_2d(&tm_a, xp, (int)wk.row0);
                    if (CG == 1) {
                        tma_prefetch_2d(&tm_b0, xp, b0);
                        tma_prefetch_2d(&tm_b1, xp, b1);
                    } else {
                        tma_prefetch_2d(tm_bh, xp, bh);
                    }
                }
                if (!mbar_wait(&empty[stage], phase ^ 1, abort_flag, p.err, p.wait_limit_ns)) { ok = false; break; }
                inflight &= ~(1u << stage);
                const bool gather_a = C::GATHER && p.a_gather != nullptr;  // the gather warps bring A
                if (rank == 0) mbar_expect_tx(&full[stage], CG * ((gather_a ? 0 : A_BYTES) + (RAW ? RAW : BH)));
                if (gather_a) {
                } else if (rank == 0) {
                    tma_load_2d(sA + stage * A_BYTES, &tm_a, kb * BK, (int)wk.row0, &full[stage]);
                } else {
                    tma_load_2d_to_pair_leader(sA + stage * A_BYTES, &tm_a, kb * BK, (int)wk.row0, &full[stage]);
                }
                // raw boxes are BK elements wide: BK bytes (fp8) or BK/2 bytes (int4, MXFP4)
                const int xr = packed4<WQ>() ? kb * (BK / 2) : kb * BK;
                if (CG == 1) {
                    if (RAW == 0) {
                        tma_load_2d(sB + stage * BH, &tm_b0, kb * BK, b0, &full[stage]);
                        tma_load_2d(sB + stage * BH + BH / 2, &tm_b1, kb * BK, b1, &full[stage]);
                    } else {
                        tma_load_2d(sR + stage * RAW, &tm_b0, xr, b0, &full[stage]);
                        tma_load_2d(sR + stage * RAW + RAW / 2, &tm_b1, xr, b1, &full[stage]);
                    }
                } else if (rank == 0) {
                    tma_load_2d(sB + stage * BH, tm_bh, kb * BK, bh, &full[stage]);
                } else {
                    tma_load_2d_to_pair_leader(sB + stage * BH, tm_bh, kb * BK, bh, &full[stage]);
                }
                inflight |= 1u << stage;
                inflight_par = (inflight_par & ~(1u << stage)) | (phase << stage);
                if (++stage == STAGES) { stage = 0; phase ^= 1; }
            }
        }
        // let every copy issued land before the CTA leaves: after a normal run
        // these phases have completed already; after an abort (here or in
        // another role) the last loads may still be in flight. The odd CTA of
        // a pair sees its copies only through the even CTA's barrier: it waits
        // for the release of those slots instead (the MMAs that read them
        // finished), which also keeps the even CTA's last arrivals on this
        // CTA's barriers before it leaves.
        for (int s = 0; s < STAGES; ++s) {
            if (!((inflight >> s) & 1u)) continue;
            if (rank == 0) drain_wait(&full[s], (inflight_par >> s) & 1u);
            if (CG == 2) drain_wait(&empty[s], (inflight_par >> s) & 1u);
        }
    } else if (warp == 1 && lane == 0 && rank == 0) {
        // ------------------------------------------------------ MMA issuer
        int stage = 0;
        uint32_t phase = 0;
        int acc = 0;
        uint32_t acc_phase = 0;
        bool ok = true;
        bool issued = false;
        for (int w = unit; w < total && ok; w += n_units) {
            if (!(CG == 1 ? mbar_wait(&tempty[acc], acc_phase ^ 1, abort_flag, p.err, p.wait_limit_ns)
                          : mbar_wait_cluster(&tempty[acc], acc_phase ^ 1, abort_flag, p.err, p.wait_limit_ns))) {
                ok = false;
                break;
            }
            tc_fence_after();
            const uint32_t d_tmem = tmem_base + (uint32_t)(acc * BN);
            for (int kb = 0; kb < nkb; ++kb) {
                if (!mbar_wait(&full[stage], phase, abort_flag, p.err, p.wait_limit_ns)) { ok = false; break; }
                if (RAW && !mbar_wait(&conv[stage], phase, abort_flag, p.err, p.wait_limit_ns)) { ok = false; break; }
                tc_fence_after();
                const uint64_t da = sw128_desc(smem_u32(sA + stage * A_BYTES));
                const uint64_t db = sw128_desc(smem_u32(sB + stage * BH));
#pragma unroll
                for (int j = 0; j < BK / 16; ++j)  // +32 bytes along K per slice
                    mma_bf16<CG>(d_tmem, da + 2 * j, db + 2 * j, (kb | j) != 0 ? 1u : 0u);
                issued = true;
                commit_to<CG>(&empty[stage], 0x3);
                if (++stage == STAGES) { stage = 0; phase ^= 1; }
            }
            if (!ok) break;
            commit_to<CG>(&tfull[acc], 0x3);
            if (++acc == 2) { acc = 0; acc_phase ^= 1; }
        }
        if (issued) {
            // every MMA issued has finished before TMEM is released (after a
            // normal run the epilogue has seen them all; after an abort in
            // another role this issuer may have run up to two tiles ahead)
            commit_to<CG>(drain, 0x1);
            drain_wait(drain, 0);
        }
    } else if (warp >= 2 && warp < 6) {
        // -------------------------------------------------------- epilogue
        const int q = warp & 3;       // TMEM lane quarter of this warp
        const int r = q * 32 + lane;  // tile row of this thread
        uint8_t* stage_buf = sE + q * 4096;  // two 2 KB buffers of this warp
        int sbuf = 0;
        int acc = 0;
        uint32_t acc_phase = 0;
        for (int w = unit; w < total; w += n_units) {
            const Work wk = decode_work<CG>(p, w, rank);
            if (!warp_wait(&tfull[acc], acc_phase, abort_flag, p.err, p.wait_limit_ns)) break;
            tc_fence_after();
            const uint32_t t_row = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * BN);
            // all 32 rows of this warp belong to the tile: one TMA store per 32 columns;
            // otherwise plain stores of the valid rows only (the rows past the tile's end
            // belong to the next expert and are written by another tile)
            const bool via_tma = L::EPI_BYTES > 0 && q * 32 + 32 <= wk.rows && p.out_f32 == nullptr && p.fuse_k == 0;
            const int col0 = p.swiglu ? wk.nt * (BN / 2) : wk.nt * BN;
            __nv_bfloat16* dst = p.out + (wk.row0 + r) * (int64_t)p.out_cols + col0;
            const bool valid = r < wk.rows;
            // fused Weight Sum: this row's pair and routing weight; the row goes to its slot (pair order)
            int64_t pair = 0;
            float wpair = 0.0f;
            if (p.fuse_k && valid) {
                pair = p.sorted_pair[wk.row0 + r];
                wpair = p.topk_w[pair];
                dst = p.out + pair * (int64_t)p.out_cols + col0;
            }
            const int ncols = p.swiglu ? BN / 2 : BN;
#pragma unroll 1
            for (int c = 0; c < ncols; c += 32) {
                float v[32];
                tmem_ld32(t_row + c, v);
                if (p.swiglu) {
                    float u[32];
                    tmem_ld32(t_row + BN / 2 + c, u);
#pragma unroll
                    for (int i = 0; i < 32; ++i) v[i] = silu_mul(v[i], u[i]);
                }
                if (via_tma) {
                    uint8_t* buf = stage_buf + sbuf * 2048;
                    if (lane == 0) bulk_wait_read<1>();  // the store that last read buf is done reading
                    __syncwarp();
                    stage_bf16x32(buf, lane, v);
                    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                    __syncwarp();
                    if (lane == 0) tma_store_2d(&tm_out, buf, col0 + c, (int)(wk.row0 + q * 32));
                    sbuf ^= 1;
                } else if (valid && p.out_f32) {
                    float* dst32 = p.out_f32 + (wk.row0 + r) * (int64_t)p.out_cols + col0 + c;
#pragma unroll
                    for (int i = 0; i < 32; ++i) {
                        const int col = col0 + c + i;
                        if (col < p.f32_cols) dst32[i] = p.col_bias ? __fadd_rn(v[i], p.col_bias[col]) : v[i];
                    }
                } else if (valid) {
                    if (p.fuse_k) {
#pragma unroll
                        for (int i = 0; i < 32; ++i) v[i] *= wpair;
                    }
                    store_bf16x32(dst + c, v);
                }
            }
            // this warp's reads of the accumulator are done: one arrival on the
            // issuing CTA's barrier (for a pair, possibly the other CTA's)
            tc_fence_before();
            __syncwarp();
            if (lane == 0) {
                if (CG == 1) mbar_arrive(&tempty[acc]);
                else mbar_arrive_rank(&tempty[acc], 0);
            }
            if (p.fuse_k) fused_weight_sum(p, valid, pair, col0);  // warp-uniform
            if (++acc == 2) { acc = 0; acc_phase ^= 1; }
        }
        if (lane == 0) bulk_wait_all();  // stores complete before the CTA exits
    } else if (RAW && warp >= 6) {
        // ------------------------------------------- weight decode (B rows)
        const int r = threadIdx.x - 6 * 32;  // B row 0 .. C::B_ROWS-1 held by this CTA
        const int half = CG == 2 ? (int)rank : r >> 7;
        const void* scales = half ? p.scale1 : p.scale0;
        const int kgroups = p.K / 128;
        int stage = 0;
        uint32_t phase = 0;
        bool ok = true;
        for (int w = unit; w < total && ok; w += n_units) {
            const Work wk = decode_work<CG>(p, w, rank);
            int b0, b1;
            b_rows(p, wk, b0, b1);
            const int64_t brow = (half ? b1 : b0) + (r & 127);  // absolute row of the stacked B tensor
            // scale entry j of this row, loaded four entries ahead so that no
            // k-block waits on a global load before decoding: for the 128-wide
            // k group j one fp32 per 128x128 block (fp8) or one bf16 per row
            // (int4); for MXFP4 the two E8M0 bytes of k-block j (as raw bits)
            constexpr int KB_PER_SCALE = WQ == GBMOE_MXFP4 ? 1 : 2;
            auto scale_of = [&](int j) -> float {
                if (j >= nkb / KB_PER_SCALE) return 0.0f;
                if (WQ == GBMOE_FP8_E4M3_B128) return static_cast<const float*>(scales)[(brow / 128) * kgroups + j];
                if (WQ == GBMOE_MXFP4)
                    return __uint_as_float(
                        *reinterpret_cast<const uint16_t*>(static_cast<const uint8_t*>(scales) + brow * (p.K / 32) + 2 * j));
                return __bfloat162float(static_cast<const __nv_bfloat16*>(scales)[brow * kgroups + j]);
            };
            float sc0 = scale_of(0), sc1 = scale_of(1), sc2 = scale_of(2), sc3 = scale_of(3);
            for (int kb = 0; kb < nkb; ++kb) {
                if (kb > 0 && kb % KB_PER_SCALE == 0) {  // next scale entry
                    sc0 = sc1; sc1 = sc2; sc2 = sc3;
                    sc3 = scale_of(kb / KB_PER_SCALE + 3);
                }
                if (!warp_wait(&full[stage], phase, abort_flag, p.err, p.wait_limit_ns)) { ok = false; break; }
                const uint8_t* raw = sR + stage * RAW;
                uint8_t* dstB = sB + stage * BH;
                if (WQ == GBMOE_FP8_E4M3_B128) {
#pragma unroll
                    for (int c = 0; c < 4; ++c) {
                        const uint4 v = *reinterpret_cast<const uint4*>(raw + sw64_off(r, c));
                        uint4 o0, o1;
                        decode_fp8_16(v, sc0, o0, o1);
                        *reinterpret_cast<uint4*>(dstB + sw128_off(r, 2 * c)) = o0;
                        *reinterpret_cast<uint4*>(dstB + sw128_off(r, 2 * c + 1)) = o1;
                    }
                } else if (WQ == GBMOE_MXFP4) {
                    const uint32_t pair = __float_as_uint(sc0);  // E8M0 of elements 0-31, 32-63
#pragma unroll
                    for (int c = 0; c < 2; ++c) {
                        const __nv_bfloat162 scv = e8m0_bf16x2((pair >> (8 * c)) & 0xffu);
                        const uint4 v = *reinterpret_cast<const uint4*>(raw + sw32_off(r, c));
                        const uint32_t ws[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
                        for (int i = 0; i < 4; ++i)
                            *reinterpret_cast<uint4*>(dstB + sw128_off(r, 4 * c + i)) = decode_mxfp4_8(ws[i], scv);
                    }
                } else {
                    const __nv_bfloat162 sc2v = __float2bfloat162_rn(sc0);  // exact: sc0 came from a bf16
#pragma unroll
                    for (int c = 0; c < 2; ++c) {
                        const uint4 v = *reinterpret_cast<const uint4*>(raw + sw32_off(r, c));
                        const uint32_t ws[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
                        for (int i = 0; i < 4; ++i)
                            *reinterpret_cast<uint4*>(dstB + sw128_off(r, 4 * c + i)) = decode_int4_8(ws[i], sc2v);
                    }
                }
                // make the generic-proxy writes visible to the tensor core, then signal
                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                __syncwarp();
                if (lane == 0) mbar_arrive(&conv[stage]);
                if (++stage == STAGES) { stage = 0; phase ^= 1; }
            }
        }
    }
    if (C::GATHER && warp >= 6 + C::CONVERT_WARPS && p.a_gather != nullptr) {
        // ----------------------------------------------- A row gather
        // warp g copies A rows 32g .. 32g+31 of each k block (64 bf16 = 128
        // bytes a row) from their x rows into the 128-byte-swizzled slot, four
        // whole rows per instruction (lane l: row 4i + l/8, 16-byte chunk l%8);
        // a warp signals a slot once its copies of it landed (GATHER_AHEAD k
        // blocks later), after a proxy fence that makes them visible to the MMAs
        constexpr int D = C::GATHER_AHEAD;
        static_assert(!C::GATHER || D < STAGES, "a gather warp must signal a slot before it needs that slot again");
        const int row_base = (warp - 6 - C::CONVERT_WARPS) * 32 + (lane >> 3);
        const int chunk = lane & 7;
        int stage = 0;
        uint32_t phase = 0;
        int64_t issued = 0;
        bool ok = true;
        for (int w = unit; w < total && ok; w += n_units) {
            const Work wk = decode_work<CG>(p, w, rank);
            const __nv_bfloat16* src[8];  // this lane's chunk of rows row_base + 4i
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const int64_t prow = wk.row0 + row_base + 4 * i;
                int32_t tok = 0;
                if (prow < p.n_rows) {
                    const int32_t sp = p.a_gather[prow];
                    tok = sp >= 0 ? sp / p.a_gather_div : 0;
                }
                src[i] = p.a_src + (int64_t)tok * p.K + 8 * chunk;
            }
            for (int kb = 0; kb < nkb; ++kb) {
                if (!warp_wait(&empty[stage], phase ^ 1, abort_flag, p.err, p.wait_limit_ns)) { ok = false; break; }
                uint8_t* dst = sA + stage * A_BYTES;
#pragma unroll
                for (int i = 0; i < 8; ++i) cp_async_16(dst + sw128_off(row_base + 4 * i, chunk), src[i] + kb * BK);
                asm volatile("cp.async.commit_group;" ::: "memory");
                if (++issued > D) {  // the k block D back has landed: signal its slot
                    asm volatile("cp.async.wait_group %0;" ::"n"(D) : "memory");
                    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&full[(stage + STAGES - D) % STAGES]);
                }
                if (++stage == STAGES) { stage = 0; phase ^= 1; }
            }
        }
        // the last k blocks' copies land before the CTA leaves; after a normal
        // run their slots are signalled too
        asm volatile("cp.async.wait_group 0;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        __syncwarp();
        if (ok && lane == 0)
            for (int64_t i = issued > D ? issued - D : 0; i < issued; ++i) mbar_arrive(&full[i % STAGES]);
    }
    tc_fence_before();
    __syncthreads();
    // a pair: neither CTA releases TMEM or leaves while the other may still
    // signal its barriers or the MMAs may still write its TMEM
    if constexpr (CG == 2) cluster_sync();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc<CG>(tmem_base);
    }
}

// ------------------------------------------------------ x rows in sorted order

__global__ void __launch_bounds__(256)
gather_rows_kernel(const uint4* __restrict__ x, const int32_t* __restrict__ sorted_pair, int pair_div,
                   int64_t n_rows, int vec_per_row, uint4* __restrict__ out) {
    pdl_enter();
    const int64_t total = n_rows * vec_per_row;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = i / vec_per_row;
        const int c = (int)(i - r * vec_per_row);
        const int32_t pr = sorted_pair[r];  // -1 past the last kept pair: a zero row
        out[i] = pr >= 0 ? x[(int64_t)(pr / pair_div) * vec_per_row + c] : make_uint4(0, 0, 0, 0);
    }
}

// ------------------------------------- one-pass decode of quantised weights

// Active experts' quantised [N, K] matrices -> bf16 [E, N, K]. A warp takes
// whole rows; lane l decodes the 8-weight pieces l, l+32, ... of the row (8
// fp8 bytes or one 32-bit word of int4 each) into 16-byte bf16 chunks, so a
// warp reads 256 or 128 contiguous bytes and writes 512 per step, with
// kDqUnroll pieces loaded ahead. The decode functions and scale handling are
// the GEMM converter warps', so the copy holds exactly the bf16 operands the
// in-GEMM decode would produce.
constexpr int kDqUnroll = 4;
constexpr int kDqWarps = 8;

template <int WQ>
__global__ void __launch_bounds__(kDqWarps * 32)
dequant_weights_kernel(const uint8_t* __restrict__ w, const void* __restrict__ s, int N, int K,
                       const int32_t* __restrict__ sched, __nv_bfloat16* __restrict__ out) {
    pdl_enter();
    const int slot = blockIdx.y;
    if (slot >= sched[0]) return;
    const int64_t e = sched[kSchedHeader + slot];
    constexpr bool kFp8 = WQ == GBMOE_FP8_E4M3_B128;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int ppr = K / 8;      // pieces per row
    const int kgroups = K / 128;
    for (int n = blockIdx.x * kDqWarps + warp; n < N; n += gridDim.x * kDqWarps) {
        const int64_t row = e * N + n;
        const uint8_t* src = w + row * (kFp8 ? K : K / 2);
        uint4* dst = reinterpret_cast<uint4*>(out + row * K);
        // scale of 128-wide k group g of this row
        const float* s8 = kFp8 ? static_cast<const float*>(s) + (e * (N / 128) + n / 128) * kgroups : nullptr;
        const __nv_bfloat16* s4 =
            WQ == GBMOE_INT4_G128 ? static_cast<const __nv_bfloat16*>(s) + row * kgroups : nullptr;
        const uint8_t* smx = WQ == GBMOE_MXFP4 ? static_cast<const uint8_t*>(s) + row * (K / 32) : nullptr;
        for (int p0 = lane; p0 < ppr; p0 += 32 * kDqUnroll) {
            uint2 raw[kDqUnroll];
#pragma unroll
            for (int u = 0; u < kDqUnroll; ++u) {
                const int pc = p0 + 32 * u;
                raw[u] = make_uint2(0, 0);
                if (pc < ppr) {
                    if constexpr (kFp8) raw[u] = __ldcs(reinterpret_cast<const uint2*>(src) + pc);
                    else raw[u].x = __ldcs(reinterpret_cast<const uint32_t*>(src) + pc);
                }
            }
#pragma unroll
            for (int u = 0; u < kDqUnroll; ++u) {
                const int pc = p0 + 32 * u;
                if (pc >= ppr) break;
                const int g = pc >> 4;  // 16 pieces of 8 per 128-wide group
                if constexpr (kFp8) {
                    uint4 o0, o1;  // decode_fp8_16 takes 16 bytes; the upper 8 are unused here
                    decode_fp8_16(make_uint4(raw[u].x, raw[u].y, 0, 0), s8[g], o0, o1);
                    dst[pc] = o0;
                } else if constexpr (WQ == GBMOE_MXFP4) {
                    dst[pc] = decode_mxfp4_8(raw[u].x, e8m0_bf16x2(smx[pc >> 2]));  // 4 pieces per 32-block
                } else {
                    dst[pc] = decode_int4_8(raw[u].x, __float2bfloat162_rn(__bfloat162float(s4[g])));
                }
            }
        }
    }
}

// ------------------------------------------------------------------- host

static bool map_bf16(CUtensorMap* m, const void* base, int64_t rows, int64_t cols) {
    return make_map(m, base, rows, cols * 2, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, BK, CU_TENSOR_MAP_SWIZZLE_128B);
}

// GEMM output [rows, cols] bf16 in {32 columns, 32 rows} boxes, 64-byte swizzle (epilogue TMA stores)
static bool map_out(CUtensorMap* m, const void* base, int64_t rows, int64_t cols) {
    return make_map(m, base, rows, cols * 2, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, 32, CU_TENSOR_MAP_SWIZZLE_64B, 32);
}

// B operand [rows, K] in the weight format WQ
static bool map_weights(CUtensorMap* m, int wq, const void* base, int64_t rows, int64_t K) {
    switch (wq) {
        case GBMOE_BF16: return map_bf16(m, base, rows, K);
        case GBMOE_FP8_E4M3_B128:
            return make_map(m, base, rows, K, CU_TENSOR_MAP_DATA_TYPE_UINT8, 1, BK, CU_TENSOR_MAP_SWIZZLE_64B);
        case GBMOE_INT4_G128:
        case GBMOE_MXFP4:
            return make_map(m, base, rows, K / 2, CU_TENSOR_MAP_DATA_TYPE_UINT8, 1, BK / 2, CU_TENSOR_MAP_SWIZZLE_32B);
        default: return false;
    }
}

template <int WQ, int CG>
static cudaError_t set_smem_attr() {
    static DeviceOnce smem_set;
    return smem_set.run([] {
        return cudaFuncSetAttribute(tc_gemm_kernel<WQ, CG>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    Layout<WQ, CG>::SMEM_BYTES);
    });
}

// CTA pairs of the CG = 2 kernel for WQ that fit on the device at once
// (queried once per device), 0 when none does
template <int WQ>
static int pair_units() {
    static std::atomic<int> cache[kMaxDevices];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return 0;
    if (const int n = cache[dev].load(std::memory_order_relaxed); n > 0) return n;
    if (set_smem_attr<WQ, 2>() != cudaSuccess) return 0;
    const int n = max_active_clusters(tc_gemm_kernel<WQ, 2>, Cfg<WQ, 2>::THREADS, Layout<WQ, 2>::SMEM_BYTES, 2);
    if (n > 0) cache[dev].store(n, std::memory_order_relaxed);
    return n;
}

template <int WQ, int CG>
static cudaError_t launch_gemm_t(const CUtensorMap& a, const CUtensorMap& b0, const CUtensorMap& b1,
                                 const CUtensorMap& out, const Params& prm, int64_t max_work, cudaStream_t stream) {
    if (const cudaError_t e = set_smem_attr<WQ, CG>(); e != cudaSuccess) return e;
    int units;  // persistent CTAs, or CTA pairs
    if constexpr (CG == 1) units = sm_count();
    else units = pair_units<WQ>();
    if (units <= 0) return cudaErrorNotSupported;
    const int grid = (int)min64(units, max_work) * CG;
    if (grid <= 0) return cudaSuccess;
    cudaError_t le;
    if (CG == 1)
        le = launch_k(tc_gemm_kernel<WQ, CG>, dim3(grid), dim3(Cfg<WQ, CG>::THREADS), Layout<WQ, CG>::SMEM_BYTES,
                      stream, a, b0, b1, out, prm);
    else
        le = launch_k_cluster(tc_gemm_kernel<WQ, CG>, dim3(grid), dim3(Cfg<WQ, CG>::THREADS),
                              Layout<WQ, CG>::SMEM_BYTES, stream, 2, a, b0, b1, out, prm);
    if (le != cudaSuccess) return le;
    return cudaGetLastError();
}

template <int CG>
static cudaError_t launch_gemm(int wq, const CUtensorMap& a, const CUtensorMap& b0, const CUtensorMap& b1,
                               const CUtensorMap& out, const Params& prm, int64_t max_work, cudaStream_t stream) {
    if constexpr (CG == 2) {
        if (wq != GBMOE_BF16) return cudaErrorNotSupported;
        return launch_gemm_t<GBMOE_BF16, 2>(a, b0, b1, out, prm, max_work, stream);
    } else {
        switch (wq) {
            case GBMOE_BF16: return launch_gemm_t<GBMOE_BF16, 1>(a, b0, b1, out, prm, max_work, stream);
            case GBMOE_FP8_E4M3_B128:
                return launch_gemm_t<GBMOE_FP8_E4M3_B128, 1>(a, b0, b1, out, prm, max_work, stream);
            case GBMOE_INT4_G128: return launch_gemm_t<GBMOE_INT4_G128, 1>(a, b0, b1, out, prm, max_work, stream);
            case GBMOE_MXFP4: return launch_gemm_t<GBMOE_MXFP4, 1>(a, b0, b1, out, prm, max_work, stream);
            default: return cudaErrorInvalidValue;
        }
    }
}

}  // namespace tc

bool ffn_tc_supported(const FfnProblem& p) {
    const bool wq_ok = p.w_dtype == GBMOE_BF16 || p.w_dtype == GBMOE_FP8_E4M3_B128 ||
                       p.w_dtype == GBMOE_INT4_G128 || p.w_dtype == GBMOE_MXFP4;
    return p.act_dtype == GBMOE_BF16 && wq_ok && p.H % 256 == 0 && p.I % 128 == 0 && tc::encode_fn() != nullptr;
}

// the CTA-pair kernel runs this problem on the current device: its B tiles
// are bf16 (bf16 weights, or a decode-once copy: w_dq set)
bool ffn_tc_pair_supported(const FfnProblem& p) {
    if (!ffn_tc_supported(p)) return false;
    if (p.w_dtype != GBMOE_BF16 && !p.w_dq) return false;
    return tc::pair_units<GBMOE_BF16>() > 0;
}

// Decodes gate, up and down of the active experts into the bf16 copy w_dq
// and returns the problem with its weights pointing there.
static cudaError_t dequant_all(const FfnProblem& p, FfnProblem& q, cudaStream_t stream) {
    using namespace tc;
    q = p;
    __nv_bfloat16* dq = static_cast<__nv_bfloat16*>(p.w_dq);
    const int64_t gu = (int64_t)p.E * p.I * p.H;
    struct Part { const void* w; const void* s; int N, K; __nv_bfloat16* out; };
    const Part parts[3] = {{p.w_gate, p.s_gate, p.I, p.H, dq}, {p.w_up, p.s_up, p.I, p.H, dq + gu},
                           {p.w_down, p.s_down, p.H, p.I, dq + 2 * gu}};
    for (const Part& pt : parts) {
        const dim3 grid((unsigned)((pt.N + kDqWarps - 1) / kDqWarps), (unsigned)p.E);
        auto kernel = p.w_dtype == GBMOE_FP8_E4M3_B128 ? dequant_weights_kernel<GBMOE_FP8_E4M3_B128>
                      : p.w_dtype == GBMOE_MXFP4        ? dequant_weights_kernel<GBMOE_MXFP4>
                                                        : dequant_weights_kernel<GBMOE_INT4_G128>;
        const cudaError_t err = launch_k(kernel, dim3(grid), dim3(kDqWarps * 32), 0, stream,
                                         static_cast<const uint8_t*>(pt.w), pt.s, pt.N, pt.K, p.sched, pt.out);
        if (err != cudaSuccess) return err;
    }
    q.w_dtype = GBMOE_BF16;
    q.w_gate = dq; q.w_up = dq + gu; q.w_down = dq + 2 * gu;
    q.s_gate = q.s_up = q.s_down = nullptr;
    q.w_dq = nullptr;
    return cudaSuccess;
}

// Router logits on the tensor cores: logits[t, e] = x[t, :] . wg[e, :]
// (+ bias[e]), x [T, H] and wg [E, H] bf16, fp32 accumulation in the tensor
// core's own order (the caller audits near ties against the fixed order).
// sched: schedule ints for one problem of T rows.
cudaError_t launch_gate_tc(const void* x, const void* wg, const float* bias, float* logits, int T, int H, int E,
                           int32_t* sched, int32_t* err, cudaStream_t stream) {
    using namespace tc;
    if (T == 0) return cudaSuccess;
    cudaError_t e = launch_ffn_schedule(nullptr, 1, T, BM, sched, stream);
    if (e != cudaSuccess) return e;
    CUtensorMap ma, mb, mo;
    // (mo is a placeholder: the fp32 epilogue stores from registers)
    if (!map_bf16(&ma, x, T, H) || !map_bf16(&mb, wg, E, H) || !map_out(&mo, x, T, H)) return cudaErrorInvalidValue;
    Params g{};
    g.K = H; g.n_tiles = (E + BN - 1) / BN; g.out_cols = E; g.b_rows_per_expert = 0; g.swiglu = 0;
    g.counts = nullptr; g.offsets = nullptr; g.sched = sched; g.E = 1; g.n_rows = T;
    g.out = nullptr; g.err = err; g.scale0 = g.scale1 = nullptr;
    g.wait_limit_ns = tc_wait_limit_ns();
    g.out_f32 = logits; g.col_bias = bias; g.f32_cols = E;
    return launch_gemm<1>(GBMOE_BF16, ma, mb, mb, mo, g, sched_max_tiles(1, T, BM) * g.n_tiles, stream);
}

cudaError_t launch_ffn_tc(const FfnProblem& pin, cudaStream_t stream) {
    using namespace tc;
    if (pin.n_rows == 0) return cudaSuccess;
    const int tile_m = pin.cta_pair ? 2 * BM : BM;  // M tile of one CTA, or of a CTA pair
    cudaError_t err = launch_ffn_schedule(pin.counts, pin.E, pin.n_rows, tile_m, pin.sched, stream);
    if (err != cudaSuccess) return err;
    FfnProblem p = pin;
    if (pin.w_dq && (pin.w_dtype == GBMOE_FP8_E4M3_B128 || pin.w_dtype == GBMOE_INT4_G128 ||
                     pin.w_dtype == GBMOE_MXFP4))
        if ((err = dequant_all(pin, p, stream)) != cudaSuccess) return err;
    // A operand of the gate/up GEMM: x rows in sorted order. The one-CTA bf16
    // GEMM gathers them from x itself; otherwise a gathered copy (x itself
    // when rows are already in order: no sorted_pair, the shared expert)
    const void* a_rows = p.x;
    const bool self_gather = p.sorted_pair && !pin.cta_pair && p.w_dtype == GBMOE_BF16;
    if (p.sorted_pair && !self_gather) {
        if (!p.x_sorted) return cudaErrorInvalidValue;  // the workspace holds no sorted copy for this route
        const int vpr = p.H * 2 / 16;
        const int64_t nvec = p.n_rows * vpr;
        const int gblocks = (int)min64((nvec + 255) / 256, (int64_t)sm_count() * 16);
        if (const cudaError_t le = launch_k(gather_rows_kernel, dim3(gblocks), dim3(256), 0, stream,
                static_cast<const uint4*>(p.x), p.sorted_pair, p.pair_div, p.n_rows, vpr,
                static_cast<uint4*>(p.x_sorted)); le != cudaSuccess)
            return le;
        if ((err = cudaGetLastError()) != cudaSuccess) return err;
        a_rows = p.x_sorted;
    }

    const int64_t max_m = sched_max_tiles(p.E, p.n_rows, tile_m);
    CUtensorMap ma, mg, mu, mh, md, oh, oy;
    // (with self_gather the A map is unused; it still spans only x's own rows)
    const int64_t a_map_rows = self_gather ? p.n_rows / p.pair_div : p.n_rows;
    if (!map_bf16(&ma, a_rows, a_map_rows, p.H) || !map_weights(&mg, p.w_dtype, p.w_gate, (int64_t)p.E * p.I, p.H) ||
        !map_weights(&mu, p.w_dtype, p.w_up, (int64_t)p.E * p.I, p.H) || !map_bf16(&mh, p.h, p.n_rows, p.I) ||
        !map_weights(&md, p.w_dtype, p.w_down, (int64_t)p.E * p.H, p.I) || !map_out(&oh, p.h, p.n_rows, p.I) ||
        !map_out(&oy, p.y, p.n_rows, p.H))
        return cudaErrorInvalidValue;

    Params g{};
    g.K = p.H; g.n_tiles = p.I / (BN / 2); g.out_cols = p.I; g.b_rows_per_expert = p.I; g.swiglu = 1;
    g.counts = p.counts; g.offsets = p.offsets; g.sched = p.sched; g.E = p.E; g.n_rows = p.n_rows;
    g.out = static_cast<__nv_bfloat16*>(p.h); g.err = p.err;
    g.scale0 = p.s_gate; g.scale1 = p.s_up;
    g.wait_limit_ns = tc_wait_limit_ns();
    if (self_gather) {
        g.a_gather = p.sorted_pair;
        g.a_gather_div = p.pair_div;
        g.a_src = static_cast<const __nv_bfloat16*>(p.x);
    }
    auto gemm = pin.cta_pair ? launch_gemm<2> : launch_gemm<1>;
    if ((err = gemm(p.w_dtype, ma, mg, mu, oh, g, max_m * g.n_tiles, stream)) != cudaSuccess) return err;

    Params d = g;
    d.a_gather = nullptr;  // the down GEMM reads h, already in sorted order
    d.K = p.I; d.n_tiles = p.H / BN; d.out_cols = p.H; d.b_rows_per_expert = p.H; d.swiglu = 0;
    d.out = static_cast<__nv_bfloat16*>(p.y);
    d.scale0 = p.s_down; d.scale1 = p.s_down;
    if (p.fuse_k) {  // Weight Sum in the down GEMM: y holds the weighted slots (pair order)
        d.fuse_k = p.fuse_k;
        d.sorted_pair = p.sorted_pair;
        d.topk_w = p.topk_w;
        d.y_shared = static_cast<const __nv_bfloat16*>(p.y_shared);
        d.out_final = static_cast<__nv_bfloat16*>(p.out_final);
        d.arrive = p.arrive;
    }
    return gemm(p.w_dtype, mh, md, md, oy, d, max_m * d.n_tiles, stream);
}

}  // namespace gbmoe
