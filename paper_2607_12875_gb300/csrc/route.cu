// MoE Gate: router logits, expert choice and routing weights.
//
// Two kernels. gate_logits computes l[t,e] = x[t,:].Wg[e,:] (+ bias[e]) in
// fp32 in the fixed order the layer's definition uses (32 partial sums over
// interleaved 8-element chunks, one fused multiply-add per element, then a
// butterfly of pairwise sums), so the expert choice is bit-identical to the
// oracle's. A warp owns TB tokens x 8 experts; lane l holds the partial sums
// of chunks l, l+32, ... for all of them, which is exactly the fixed order.
// select_experts then runs one warp per token over the logits. Large batches
// use a shared-memory-staged variant with the same order (below).
#include "common.cuh"
#include "kernels.h"

namespace gbmoe {

constexpr int kGateWarps = 8;
constexpr int kGateExpertsPerWarp = 8;

template <typename TA, int TB>
__global__ void __launch_bounds__(kGateWarps * 32)
gate_logits_kernel(const TA* __restrict__ x, const TA* __restrict__ wg, const float* __restrict__ bias,
                   float* __restrict__ logits, int T, int H, int E) {
    pdl_enter();
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int t0 = blockIdx.x * TB;
    const int e0 = (blockIdx.y * kGateWarps + warp) * kGateExpertsPerWarp;
    if (e0 >= E) return;
    float acc[TB][kGateExpertsPerWarp];
#pragma unroll
    for (int a = 0; a < TB; ++a)
#pragma unroll
        for (int b = 0; b < kGateExpertsPerWarp; ++b) acc[a][b] = 0.0f;

    const int nchunk = H / 8;  // H % 256 == 0: every lane gets H/256 chunks
    // two steps per iteration: their loads are in flight together (each
    // accumulator still takes its chunks in increasing order)
#pragma unroll 2
    for (int c = lane; c < nchunk; c += 32) {
        float xv[TB][8];
#pragma unroll
        for (int a = 0; a < TB; ++a) {
            int t = t0 + a;
            if (t < T) {
                Vec8<TA>::load(x + (size_t)t * H + 8 * c, xv[a]);
            } else {
#pragma unroll
                for (int i = 0; i < 8; ++i) xv[a][i] = 0.0f;
            }
        }
#pragma unroll
        for (int b = 0; b < kGateExpertsPerWarp; ++b) {
            int e = e0 + b;
            float wv[8];
            if (e < E) {
                Vec8<TA>::load(wg + (size_t)e * H + 8 * c, wv);
            } else {
#pragma unroll
                for (int i = 0; i < 8; ++i) wv[i] = 0.0f;
            }
#pragma unroll
            for (int a = 0; a < TB; ++a)
#pragma unroll
                for (int i = 0; i < 8; ++i) acc[a][b] = __fmaf_rn(xv[a][i], wv[i], acc[a][b]);
        }
    }
    // butterfly: s[p] <- s[p] + s[p ^ d], d = 16 .. 1 (one commutative add: all lanes end equal)
#pragma unroll
    for (int a = 0; a < TB; ++a)
#pragma unroll
        for (int b = 0; b < kGateExpertsPerWarp; ++b) {
            float v = acc[a][b];
#pragma unroll
            for (int d = 16; d >= 1; d >>= 1) v = __fadd_rn(v, __shfl_xor_sync(0xffffffffu, v, d));
            acc[a][b] = v;
        }
#pragma unroll
    for (int a = 0; a < TB; ++a)
#pragma unroll
        for (int b = 0; b < kGateExpertsPerWarp; ++b) {
            int t = t0 + a, e = e0 + b;
            if (lane == ((a * kGateExpertsPerWarp + b) & 31) && t < T && e < E) {
                float l = acc[a][b];
                if (bias) l = __fadd_rn(l, bias[e]);
                logits[(size_t)t * E + e] = l;
            }
        }
}

// Large batches: the same fixed order, as a CUDA-core GEMM. A CTA owns 32
// tokens x 16 experts; 256-element slabs of x and Wg go through a 3-stage
// cp.async ring in shared memory, and warp w (of 8) accumulates tokens
// 8*(w%4).. x experts 8*(w/4).. in registers. Lane l reads 8-element chunk l
// of every slab, i.e. chunks l, l+32, ... in increasing order, elements in
// increasing order inside a chunk, exactly as in the definition.
constexpr int kGT = 32, kGE = 16, kSlab = 256, kGStages = 3;
constexpr size_t kGateTiledSmem = (size_t)kGStages * (kGT + kGE) * kSlab * 2;

__device__ __forceinline__ void cp_async16(void* dst, const void* src, bool valid) {
    const uint32_t d = static_cast<uint32_t>(__cvta_generic_to_shared(dst));
    const int n = valid ? 16 : 0;  // 0 bytes read: the 16 bytes are zero-filled
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(d), "l"(src), "r"(n) : "memory");
}

__global__ void __launch_bounds__(256, 1)
gate_logits_tiled_kernel(const __nv_bfloat16* __restrict__ x, const __nv_bfloat16* __restrict__ wg,
                         const float* __restrict__ bias, float* __restrict__ logits, int T, int H, int E) {
    pdl_enter();
    extern __shared__ __align__(16) uint8_t smem[];
    uint8_t* sx = smem;                                          // [stage][kGT][kSlab] bf16
    uint8_t* sw = smem + (size_t)kGStages * kGT * kSlab * 2;     // [stage][kGE][kSlab] bf16
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int t0 = blockIdx.x * kGT, e0 = blockIdx.y * kGE;
    const int nslab = H / kSlab;

    auto load_slab = [&](int j) {
        const int st = j % kGStages;
        // x: kGT rows x 32 chunks; Wg: kGE rows x 32 chunks; 16 bytes each
        for (int i = threadIdx.x; i < (kGT + kGE) * 32; i += 256) {
            const int row = i >> 5, c = i & 31;
            if (row < kGT) {
                const int t = t0 + row;
                const bool ok = t < T;
                cp_async16(sx + (((size_t)st * kGT + row) * kSlab + 8 * c) * 2,
                           x + (size_t)(ok ? t : 0) * H + (size_t)j * kSlab + 8 * c, ok);
            } else {
                const int r = row - kGT, e = e0 + r;
                const bool ok = e < E;
                cp_async16(sw + (((size_t)st * kGE + r) * kSlab + 8 * c) * 2,
                           wg + (size_t)(ok ? e : 0) * H + (size_t)j * kSlab + 8 * c, ok);
            }
        }
    };

    float acc[8][8];
#pragma unroll
    for (int a = 0; a < 8; ++a)
#pragma unroll
        for (int b = 0; b < 8; ++b) acc[a][b] = 0.0f;
    const int tg = (warp & 3) * 8, eg = (warp >> 2) * 8;

#pragma unroll
    for (int j = 0; j < kGStages - 1; ++j) {
        if (j < nslab) load_slab(j);
        asm volatile("cp.async.commit_group;" ::: "memory");
    }
    for (int j = 0; j < nslab; ++j) {
        asm volatile("cp.async.wait_group %0;" ::"n"(kGStages - 2) : "memory");
        __syncthreads();
        if (j + kGStages - 1 < nslab) load_slab(j + kGStages - 1);
        asm volatile("cp.async.commit_group;" ::: "memory");
        const int st = j % kGStages;
        uint4 xr[8], wr[8];
#pragma unroll
        for (int a = 0; a < 8; ++a)
            xr[a] = *reinterpret_cast<const uint4*>(sx + (((size_t)st * kGT + tg + a) * kSlab + 8 * lane) * 2);
#pragma unroll
        for (int b = 0; b < 8; ++b)
            wr[b] = *reinterpret_cast<const uint4*>(sw + (((size_t)st * kGE + eg + b) * kSlab + 8 * lane) * 2);
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            float xf[8], wf[8];
#pragma unroll
            for (int a = 0; a < 8; ++a) {
                const uint32_t u = (&xr[a].x)[i >> 1];
                xf[a] = (i & 1) ? bf16hi(u) : bf16lo(u);
            }
#pragma unroll
            for (int b = 0; b < 8; ++b) {
                const uint32_t u = (&wr[b].x)[i >> 1];
                wf[b] = (i & 1) ? bf16hi(u) : bf16lo(u);
            }
#pragma unroll
            for (int a = 0; a < 8; ++a)
#pragma unroll
                for (int b = 0; b < 8; ++b) acc[a][b] = __fmaf_rn(xf[a], wf[b], acc[a][b]);
        }
    }
    asm volatile("cp.async.wait_group 0;" ::: "memory");
    // butterfly: s[p] <- s[p] + s[p ^ d], d = 16 .. 1
#pragma unroll
    for (int a = 0; a < 8; ++a)
#pragma unroll
        for (int b = 0; b < 8; ++b) {
            float v = acc[a][b];
#pragma unroll
            for (int d = 16; d >= 1; d >>= 1) v = __fadd_rn(v, __shfl_xor_sync(0xffffffffu, v, d));
            acc[a][b] = v;
        }
#pragma unroll
    for (int a = 0; a < 8; ++a)
#pragma unroll
        for (int b = 0; b < 8; ++b) {
            const int t = t0 + tg + a, e = e0 + eg + b;
            if (lane == ((a * 8 + b) & 31) && t < T && e < E) {
                float l = acc[a][b];
                if (bias) l = __fadd_rn(l, bias[e]);
                logits[(size_t)t * E + e] = l;
            }
        }
}

// ------------------------------------------------------- expert choice

// Fixed fp32 exponential for the sigmoid score (the expert choice depends on
// its exact bits, so it is not left to a library): NaN is returned as it
// is, anything else clamped to [-86, 88];
// n = rint(x*log2 e); r = (x - n*ln2_hi) - n*ln2_lo with ln2_hi the leading
// 16 bits of ln 2 (Cody-Waite reduction, exact n*ln2_hi); exp(r) from its
// degree-8 Taylor polynomial by Horner's rule, a separate rounded multiply
// and add per step; times 2^n assembled from exponent bits.
__device__ __forceinline__ float pinned_exp(float x) {
    const float kLog2e = __uint_as_float(0x3fb8aa3bu);  // fp32(1/ln 2)
    const float kLn2Hi = __uint_as_float(0x3f317200u);  // 0.693145751953125
    const float kLn2Lo = __uint_as_float(0x35bfbe8eu);  // fp32(ln 2 - kLn2Hi)
    const uint32_t kInvFact[9] = {0x3f800000u, 0x3f800000u, 0x3f000000u, 0x3e2aaaabu, 0x3d2aaaabu,
                                  0x3c088889u, 0x3ab60b61u, 0x39500d01u, 0x37d00d01u};  // fp32(1/i!)
    if (x != x) return x;  // NaN in, NaN out
    x = fminf(fmaxf(x, -86.0f), 88.0f);
    float n = rintf(__fmul_rn(x, kLog2e));
    float r = __fsub_rn(x, __fmul_rn(n, kLn2Hi));
    r = __fsub_rn(r, __fmul_rn(n, kLn2Lo));
    float p = __uint_as_float(kInvFact[8]);
#pragma unroll
    for (int i = 7; i >= 0; --i) p = __fadd_rn(__fmul_rn(p, r), __uint_as_float(kInvFact[i]));
    return __fmul_rn(p, __uint_as_float((uint32_t)((int)n + 127) << 23));
}

__device__ __forceinline__ float pinned_sigmoid(float l) {
    return __fdiv_rn(1.0f, __fadd_rn(1.0f, pinned_exp(-l)));
}

// (key, index) with "larger key, then smaller index" as the better candidate.
// Keys are never NaN here (choice_key), so this is a strict total order, and
// a real candidate (index < kNone) beats an empty one even at key -inf.
constexpr int kNone = 0x7fffffff;
__device__ __forceinline__ bool better(float ka, int ia, float kb, int ib) {
    return ka > kb || (ka == kb && ia < ib);
}

// Key a score takes in the expert choice: a NaN counts as -infinity, so
// non-finite logits still give valid, deterministic ids (ties to the lower index).
__device__ __forceinline__ float choice_key(float v) { return v != v ? -INFINITY : v; }

__device__ __forceinline__ void warp_best(float& k, int& i) {
#pragma unroll
    for (int d = 16; d >= 1; d >>= 1) {
        float ko = __shfl_xor_sync(0xffffffffu, k, d);
        int io = __shfl_xor_sync(0xffffffffu, i, d);
        if (better(ko, io, k, i)) { k = ko; i = io; }
    }
}

constexpr int kSelWarps = 4;
constexpr int kMaxE = 512;

// One warp per token. Expert e lives in lane e % 32, slot e / 32.
__global__ void __launch_bounds__(kSelWarps * 32)
select_experts_kernel(const float* __restrict__ logits, const float* __restrict__ select_bias,
                      int32_t* __restrict__ topk_ids, float* __restrict__ topk_w, RouteParams rp) {
    pdl_enter();
    __shared__ float s_key[kSelWarps][kMaxE];
    __shared__ float s_sig[kSelWarps][kMaxE];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int t = blockIdx.x * kSelWarps + warp;
    if (t >= rp.T) return;
    const int E = rp.E, k = rp.top_k;
    const float* l = logits + (size_t)t * E;
    float* key = s_key[warp];
    float* sig = s_sig[warp];
    const bool sigmoid = rp.score == GBMOE_SIGMOID;
    for (int e = lane; e < E; e += 32) {
        float v = l[e];
        if (sigmoid) {
            float s = pinned_sigmoid(v);
            sig[e] = s;
            v = select_bias ? __fadd_rn(s, select_bias[e]) : s;
        }
        key[e] = choice_key(v);
    }
    __syncwarp();

    // groups kept (bit g set); all experts allowed without group limiting
    uint32_t kept = 0xffffffffu;
    const int G = sigmoid ? rp.n_group : 1;
    if (G > 1) {
        const int gs = E / G;
        float gscore = -INFINITY;
        if (lane < G) {
            float a = -INFINITY, b = -INFINITY;  // two largest q of group `lane`
            for (int e = lane * gs; e < (lane + 1) * gs; ++e) {
                float v = key[e];
                if (v > a) { b = a; a = v; } else if (v > b) { b = v; }
            }
            gscore = choice_key(__fadd_rn(a, b));  // inf + -inf is NaN
        }
        kept = 0u;
        bool taken = false;
        for (int r = 0; r < rp.topk_group; ++r) {
            float kk = (lane < G && !taken) ? gscore : -INFINITY;
            int ii = (lane < G && !taken) ? lane : kNone;
            warp_best(kk, ii);
            if (ii < 32) kept |= 1u << ii;  // always: topk_group <= G groups hold candidates
            if (lane == ii) taken = true;
        }
    }
    const int gs = E / G;

    // top-k over allowed experts, descending key, ties to the lower index
    uint32_t used = 0u;  // bit s: expert lane + 32 s already chosen
    int sel_id = 0;
    float top_key = 0.0f;
    for (int j = 0; j < k; ++j) {
        float kk = -INFINITY;
        int ii = kNone;
        for (int s = 0, e = lane; e < E; ++s, e += 32) {
            if ((used >> s) & 1u) continue;
            if (!((kept >> (e / gs)) & 1u)) continue;
            float v = key[e];
            if (ii == kNone || better(v, e, kk, ii)) { kk = v; ii = e; }
        }
        warp_best(kk, ii);
        // ii < E always (check_config keeps top_k within the kept groups' experts)
        if (ii < E && (ii & 31) == lane) used |= 1u << (ii >> 5);
        if (j == 0) top_key = kk;
        if (lane == j) sel_id = ii < E ? ii : 0;
    }

    // routing weights (lane j < k holds slot j)
    float w = 0.0f;
    if (!sigmoid) {
        float lj = (lane < k) ? l[sel_id] : 0.0f;
        float m = top_key, z = 0.0f;
        if (!rp.renormalize) {
            float mm = -INFINITY;
            for (int e = lane; e < E; e += 32) mm = fmaxf(mm, l[e]);
#pragma unroll
            for (int d = 16; d >= 1; d >>= 1) mm = fmaxf(mm, __shfl_xor_sync(0xffffffffu, mm, d));
            m = mm;
            for (int e = lane; e < E; e += 32) z += expf(l[e] - m);
        } else {
            z = (lane < k) ? expf(lj - m) : 0.0f;
        }
#pragma unroll
        for (int d = 16; d >= 1; d >>= 1) z += __shfl_xor_sync(0xffffffffu, z, d);
        w = (lane < k) ? expf(lj - m) / z * rp.routed_scale : 0.0f;
    } else {
        float sj = (lane < k) ? sig[sel_id] : 0.0f;
        float z = sj;
#pragma unroll
        for (int d = 16; d >= 1; d >>= 1) z += __shfl_xor_sync(0xffffffffu, z, d);
        w = (rp.renormalize ? sj / z : sj) * rp.routed_scale;
    }
    if (lane < k) {
        topk_ids[(size_t)t * k + lane] = sel_id;
        topk_w[(size_t)t * k + lane] = w;
    }
}

cudaError_t launch_route(const RouteParams& rp, const void* x, const void* wg, const float* logit_bias,
                         const float* select_bias, float* logits, int32_t* topk_ids, float* topk_w,
                         cudaStream_t stream) {
    if (rp.T == 0) return cudaSuccess;
    const int ey = (rp.E + kGateWarps * kGateExpertsPerWarp - 1) / (kGateWarps * kGateExpertsPerWarp);
    dim3 block(kGateWarps * 32);
    if (rp.act_dtype == GBMOE_BF16) {
        auto xp = static_cast<const __nv_bfloat16*>(x);
        auto wp = static_cast<const __nv_bfloat16*>(wg);
        if (rp.T >= 1024) {
            static DeviceOnce smem_set;
            cudaError_t e = smem_set.run([] {
                return cudaFuncSetAttribute(gate_logits_tiled_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                            (int)kGateTiledSmem);
            });
            if (e != cudaSuccess) return e;
            dim3 grid((rp.T + kGT - 1) / kGT, (rp.E + kGE - 1) / kGE);
            if (const cudaError_t le = launch_k(gate_logits_tiled_kernel, dim3(grid), dim3(256), kGateTiledSmem,
                    stream, xp, wp, logit_bias, logits, rp.T, rp.H, rp.E); le != cudaSuccess)
                return le;
        } else {
            dim3 grid((rp.T + 1) / 2, ey);
            if (const cudaError_t le = launch_k(gate_logits_kernel<__nv_bfloat16, 2>, dim3(grid), dim3(block), 0,
                    stream, xp, wp, logit_bias, logits, rp.T, rp.H, rp.E); le != cudaSuccess)
                return le;
        }
    } else {
        auto xp = static_cast<const float*>(x);
        auto wp = static_cast<const float*>(wg);
        dim3 grid((rp.T + 1) / 2, ey);
        if (const cudaError_t le = launch_k(gate_logits_kernel<float, 2>, dim3(grid), dim3(block), 0, stream, xp,
                wp, logit_bias, logits, rp.T, rp.H, rp.E); le != cudaSuccess)
            return le;
    }
    cudaError_t err = cudaGetLastError();
    if (err != cudaSuccess) return err;
    if (const cudaError_t le = launch_k(select_experts_kernel, dim3((rp.T + kSelWarps - 1) / kSelWarps),
            dim3(kSelWarps * 32), 0, stream, logits, select_bias, topk_ids, topk_w, rp); le != cudaSuccess)
        return le;
    return cudaGetLastError();
}

}  // namespace gbmoe
