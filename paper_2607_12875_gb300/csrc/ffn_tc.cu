// Fused MoE on tensor cores: grouped GEMMs with tcgen05, TMEM and TMA.
//
// Rows of each expert are contiguous after the permutation (the gate/up
// GEMM reads a gathered copy of x in sorted order, the down GEMM reads h),
// so every M tile is a plain 128-row box of a 2-D tensor. A tile that runs
// past its expert's last row reads the next expert's rows (or TMA's zero
// fill past the end); those rows are computed and never stored.
//
// One persistent CTA per SM walks the (M tile, N tile) work list built on the
// device. Warp roles (192 threads):
//   warp 0    one lane issues TMA loads of A (128 x 64) and B (2 x 128 x 64)
//             bf16 boxes, 128-byte swizzled, into a 4-stage shared ring;
//   warp 1    allocates 512 TMEM columns (two 128 x 256 fp32 accumulators)
//             and one lane issues tcgen05.mma (M=128, N=256, K=16) per
//             16-wide slice, releasing ring slots and accumulators through
//             tcgen05.commit -> mbarrier;
//   warps 2-5 read the accumulator with tcgen05.ld (warp w owns TMEM lanes
//             32*(w%4)..+31, i.e. tile rows) and write bf16 results:
//             h = silu(gate) * up for the gate/up GEMM (B rows 0-127 are the
//             gate rows, 128-255 the up rows of the same 128 columns), plain
//             y for the down GEMM.
// Every mbarrier wait is bounded (about two seconds); on expiry the CTA sets
// the device error word, stops issuing work, drains what it issued and
// frees its TMEM.
#include <cuda.h>

#include "common.cuh"
#include "ffn_sched.h"
#include "kernels.h"

namespace gbmoe {
namespace tc {

constexpr int BM = 128, BN = 256, BK = 64;  // BK bf16 = 128 bytes = one swizzle row
constexpr int STAGES = 4;
constexpr int A_BYTES = BM * BK * 2;
constexpr int B_BYTES = BN * BK * 2;
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int TMEM_COLS = 512;
constexpr int NUM_THREADS = 192;
constexpr int NUM_BARS = 2 * STAGES + 4 + 1;
constexpr int SMEM_BYTES = 1024 + STAGES * STAGE_BYTES + NUM_BARS * 8 + 16;
constexpr unsigned long long kWaitLimitNs = 2000000000ull;

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
};

// ------------------------------------------------------------ PTX wrappers

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}

__device__ __forceinline__ uint64_t global_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// Bounded wait for the phase of `bar` with the given parity. Returns false
// (after flagging the CTA and the device error word) when the limit expires
// or another role of this CTA has already given up.
__device__ __noinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag, int32_t* err) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = global_ns();
    for (uint32_t i = 1;; ++i) {
        if (mbar_try_wait(bar, parity)) return true;
        if (*abort_flag) return false;
        if ((i & 255u) == 0 && global_ns() - t0 > kWaitLimitNs) {
            *abort_flag = 1;
            set_error(err, kErrTimeout);
            return false;
        }
    }
}

__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, int x, int y, uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];"
        ::"r"(smem_u32(dst)), "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_u32(bar))
        : "memory");
}

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// Shared-memory matrix descriptor of a K-major tile stored as TMA writes it
// with 128-byte swizzling: rows of 128 bytes, 8-row groups 1024 bytes apart.
//   bits  0-13 start address >> 4      bits 16-29 leading offset >> 4 (unused here)
//   bits 32-45 stride offset >> 4      bits 46-47 descriptor version (1)
//   bits 61-63 swizzle mode (2 = 128-byte)
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
    uint64_t d = 0;
    d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
    d |= (uint64_t)1 << 16;
    d |= (uint64_t)(1024 >> 4) << 32;
    d |= (uint64_t)1 << 46;
    d |= (uint64_t)2 << 61;
    return d;
}

// Instruction descriptor, kind::f16: fp32 accumulator (bits 4-5 = 1), bf16 A
// and B (bits 7-9, 10-12 = 1), both K-major, N/8 in bits 17-22, M/16 in 24-28.
constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(BN >> 3) << 17) |
                            ((uint32_t)(BM >> 4) << 24);

__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(a_desc), "l"(b_desc), "r"(kIdesc), "r"(accumulate)
        : "memory");
}

__device__ __forceinline__ void mma_commit(uint64_t* bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
                 : "memory");
}

// 32 consecutive fp32 columns of this thread's TMEM lane
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
        "%15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
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

// ------------------------------------------------------------------ kernel

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

__global__ void __launch_bounds__(NUM_THREADS, 1)
tc_gemm_kernel(const __grid_constant__ CUtensorMap tm_a, const __grid_constant__ CUtensorMap tm_b0,
               const __grid_constant__ CUtensorMap tm_b1, const Params p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    uint8_t* sA = smem;
    uint8_t* sB = smem + STAGES * A_BYTES;
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE_BYTES);
    uint64_t* full = bars;
    uint64_t* empty = bars + STAGES;
    uint64_t* tfull = bars + 2 * STAGES;
    uint64_t* tempty = bars + 2 * STAGES + 2;
    uint64_t* drain = bars + 2 * STAGES + 4;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + NUM_BARS);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(&tfull[a], 1);
            mbar_init(&tempty[a], 4 * 32);
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
            const int b0 = wk.e * p.b_rows_per_expert + (p.swiglu ? wk.nt * (BN / 2) : wk.nt * BN);
            const int b1 = p.swiglu ? b0 : b0 + BN / 2;
            for (int kb = 0; kb < nkb; ++kb) {
                if (!mbar_wait(&empty[stage], phase ^ 1, abort_flag, p.err)) { ok = false; break; }
                inflight &= ~(1u << stage);
                mbar_expect_tx(&full[stage], STAGE_BYTES);
                tma_load_2d(sA + stage * A_BYTES, &tm_a, kb * BK, (int)wk.row0, &full[stage]);
                tma_load_2d(sB + stage * B_BYTES, &tm_b0, kb * BK, b0, &full[stage]);
                tma_load_2d(sB + stage * B_BYTES + B_BYTES / 2, &tm_b1, kb * BK, b1, &full[stage]);
                inflight |= 1u << stage;
                inflight_par = (inflight_par & ~(1u << stage)) | (phase << stage);
                if (++stage == STAGES) { stage = 0; phase ^= 1; }
            }
        }
        if (!ok) {
            // let the copies already issued land before the CTA leaves
            for (int s = 0; s < STAGES; ++s) {
                if (!((inflight >> s) & 1u)) continue;
                const uint64_t t0 = global_ns();
                while (!mbar_try_wait(&full[s], (inflight_par >> s) & 1u) && global_ns() - t0 < kWaitLimitNs) {
                }
            }
        }
    } else if (warp == 1 && lane == 0) {
        // ------------------------------------------------------ MMA issuer
        int stage = 0;
        uint32_t phase = 0;
        int acc = 0;
        uint32_t acc_phase = 0;
        bool ok = true;
        bool issued = false;
        for (int w = blockIdx.x; w < total && ok; w += gridDim.x) {
            if (!mbar_wait(&tempty[acc], acc_phase ^ 1, abort_flag, p.err)) { ok = false; break; }
            tc_fence_after();
            const uint32_t d_tmem = tmem_base + (uint32_t)(acc * BN);
            for (int kb = 0; kb < nkb; ++kb) {
                if (!mbar_wait(&full[stage], phase, abort_flag, p.err)) { ok = false; break; }
                tc_fence_after();
                const uint64_t da = sw128_desc(smem_u32(sA + stage * A_BYTES));
                const uint64_t db = sw128_desc(smem_u32(sB + stage * B_BYTES));
#pragma unroll
                for (int j = 0; j < BK / 16; ++j)  // +32 bytes along K per slice
                    mma_bf16(d_tmem, da + 2 * j, db + 2 * j, (kb | j) != 0 ? 1u : 0u);
                issued = true;
                mma_commit(&empty[stage]);
                if (++stage == STAGES) { stage = 0; phase ^= 1; }
            }
            if (!ok) break;
            mma_commit(&tfull[acc]);
            if (++acc == 2) { acc = 0; acc_phase ^= 1; }
        }
        if (!ok && issued) {
            // wait for the MMAs already issued before TMEM is released
            mma_commit(drain);
            const uint64_t t0 = global_ns();
            while (!mbar_try_wait(drain, 0) && global_ns() - t0 < kWaitLimitNs) {
            }
        }
    } else if (warp >= 2) {
        // -------------------------------------------------------- epilogue
        const int q = warp & 3;  // TMEM lane quarter of this warp
        const int r = q * 32 + lane;  // tile row of this thread
        int acc = 0;
        uint32_t acc_phase = 0;
        for (int w = blockIdx.x; w < total; w += gridDim.x) {
            const Work wk = decode_work(p, w);
            if (!mbar_wait(&tfull[acc], acc_phase, abort_flag, p.err)) break;
            tc_fence_after();
            const uint32_t t_row = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * BN);
            const bool valid = r < wk.rows;
            __nv_bfloat16* dst = p.out + (wk.row0 + r) * (int64_t)p.out_cols;
            if (p.swiglu) {
                dst += wk.nt * (BN / 2);
#pragma unroll 1
                for (int c = 0; c < BN / 2; c += 32) {
                    float g[32], u[32];
                    tmem_ld32(t_row + c, g);
                    tmem_ld32(t_row + BN / 2 + c, u);
#pragma unroll
                    for (int i = 0; i < 32; ++i) g[i] = silu_mul(g[i], u[i]);
                    if (valid) store_bf16x32(dst + c, g);
                }
            } else {
                dst += wk.nt * BN;
#pragma unroll 1
                for (int c = 0; c < BN; c += 32) {
                    float v[32];
                    tmem_ld32(t_row + c, v);
                    if (valid) store_bf16x32(dst + c, v);
                }
            }
            tc_fence_before();
            mbar_arrive(&tempty[acc]);
            if (++acc == 2) { acc = 0; acc_phase ^= 1; }
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

// ------------------------------------------------------ x rows in sorted order

__global__ void __launch_bounds__(256)
gather_rows_kernel(const uint4* __restrict__ x, const int32_t* __restrict__ sorted_pair, int pair_div,
                   int64_t n_rows, int vec_per_row, uint4* __restrict__ out) {
    const int64_t total = n_rows * vec_per_row;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = i / vec_per_row;
        const int c = (int)(i - r * vec_per_row);
        const int64_t src = sorted_pair[r] / pair_div;
        out[i] = x[src * vec_per_row + c];
    }
}

// ------------------------------------------------------------------- host

using EncodeTiled = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                 const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                 CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiled encode_fn() {
    static EncodeTiled fn = nullptr;
    static bool tried = false;
    if (!tried) {
        tried = true;
        void* ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiled>(ptr);
    }
    return fn;
}

// bf16 matrix [rows, cols] row-major; boxes of 64 columns x 128 rows, 128-byte swizzle
static bool make_map(CUtensorMap* m, const void* base, int64_t rows, int64_t cols) {
    EncodeTiled fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
    cuuint32_t box[2] = {BK, 128};
    cuuint32_t estr[2] = {1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

static int num_sms() {
    int dev = 0, n = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    return n > 0 ? n : 1;
}

static cudaError_t launch_gemm(const CUtensorMap& a, const CUtensorMap& b0, const CUtensorMap& b1, const Params& prm,
                               int64_t max_work, cudaStream_t stream) {
    static bool attr_set = false;
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(tc_gemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    const int grid = (int)min64(num_sms(), max_work);
    if (grid <= 0) return cudaSuccess;
    tc_gemm_kernel<<<grid, NUM_THREADS, SMEM_BYTES, stream>>>(a, b0, b1, prm);
    return cudaGetLastError();
}

}  // namespace tc

bool ffn_tc_supported(const FfnProblem& p) {
    return p.act_dtype == GBMOE_BF16 && p.w_dtype == GBMOE_BF16 && p.H % 256 == 0 && p.I % 128 == 0 &&
           tc::encode_fn() != nullptr;
}

cudaError_t launch_ffn_tc(const FfnProblem& p, cudaStream_t stream) {
    using namespace tc;
    if (p.n_rows == 0) return cudaSuccess;
    cudaError_t err = launch_ffn_schedule(p.counts, p.E, p.n_rows, BM, p.sched, stream);
    if (err != cudaSuccess) return err;
    // x rows in sorted order
    const int vpr = p.H * 2 / 16;
    const int64_t nvec = p.n_rows * vpr;
    const int gblocks = (int)min64((nvec + 255) / 256, 152 * 16);
    gather_rows_kernel<<<gblocks, 256, 0, stream>>>(static_cast<const uint4*>(p.x), p.sorted_pair, p.pair_div,
                                                    p.n_rows, vpr, static_cast<uint4*>(p.x_sorted));
    if ((err = cudaGetLastError()) != cudaSuccess) return err;

    const int64_t max_m = sched_max_tiles(p.E, p.n_rows, BM);
    CUtensorMap ma, mg, mu, mh, md;
    if (!make_map(&ma, p.x_sorted, p.n_rows, p.H) || !make_map(&mg, p.w_gate, (int64_t)p.E * p.I, p.H) ||
        !make_map(&mu, p.w_up, (int64_t)p.E * p.I, p.H) || !make_map(&mh, p.h, p.n_rows, p.I) ||
        !make_map(&md, p.w_down, (int64_t)p.E * p.H, p.I))
        return cudaErrorInvalidValue;

    Params g{};
    g.K = p.H; g.n_tiles = p.I / (BN / 2); g.out_cols = p.I; g.b_rows_per_expert = p.I; g.swiglu = 1;
    g.counts = p.counts; g.offsets = p.offsets; g.sched = p.sched; g.E = p.E; g.n_rows = p.n_rows;
    g.out = static_cast<__nv_bfloat16*>(p.h); g.err = p.err;
    if ((err = launch_gemm(ma, mg, mu, g, max_m * g.n_tiles, stream)) != cudaSuccess) return err;

    Params d = g;
    d.K = p.I; d.n_tiles = p.H / BN; d.out_cols = p.H; d.b_rows_per_expert = p.H; d.swiglu = 0;
    d.out = static_cast<__nv_bfloat16*>(p.y);
    return launch_gemm(mh, md, md, d, max_m * d.n_tiles, stream);
}

}  // namespace gbmoe
