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
#include <cstdlib>

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

// With a token list, tile rows are the listed tokens (list[0 .. *n_list)),
// and tiles past the list's end return at once.
__global__ void __launch_bounds__(256, 1)
gate_logits_tiled_kernel(const __nv_bfloat16* __restrict__ x, const __nv_bfloat16* __restrict__ wg,
                         const float* __restrict__ bias, float* __restrict__ logits, int T, int H, int E,
                         const int32_t* __restrict__ list, const int32_t* __restrict__ n_list) {
    pdl_enter();
    const int n_rows = list ? *n_list : T;
    if ((int)blockIdx.x * kGT >= n_rows) return;
    // token of tile row i (or -1 past the end)
    auto token = [&](int i) -> int {
        const int r = (int)blockIdx.x * kGT + i;
        return r < n_rows ? (list ? list[r] : r) : -1;
    };
    extern __shared__ __align__(16) uint8_t smem[];
    uint8_t* sx = smem;                                          // [stage][kGT][kSlab] bf16
    uint8_t* sw = smem + (size_t)kGStages * kGT * kSlab * 2;     // [stage][kGE][kSlab] bf16
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int e0 = blockIdx.y * kGE;
    const int nslab = H / kSlab;

    auto load_slab = [&](int j) {
        const int st = j % kGStages;
        // x: kGT rows x 32 chunks; Wg: kGE rows x 32 chunks; 16 bytes each
        for (int i = threadIdx.x; i < (kGT + kGE) * 32; i += 256) {
            const int row = i >> 5, c = i & 31;
            if (row < kGT) {
                const int t = token(row);
                const bool ok = t >= 0;
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
            const int t = token(tg + a), e = e0 + eg + b;
            if (lane == ((a * 8 + b) & 31) && t >= 0 && e < E) {
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

// Audit of router logits computed on the tensor cores (their fp32 sums run in
// the hardware's own order, not the fixed order of the definition). Those
// logits differ from the fixed-order ones by at most about
// scale * ||x_t|| * ||w_e|| (|sum of the same products in two orders|), so an
// expert choice whose every deciding comparison clears twice that bound is the
// fixed-order choice; any other token is recomputed in the fixed order.
struct GateAudit {
    const __nv_bfloat16* x;   // [T, H]; null: logits are fixed-order already (no audit)
    const float* wnorm_max;   // max_e ||wg[e]||_2 (one float)
    float scale;              // bound on |tensor-core logit - fixed-order logit| / (||x_t|| * max ||w_e||)
    int32_t* flagged;         // [T] tokens whose choice is too close to call (their logits are recomputed)
    int32_t* n_flagged;       // their count
};

// One warp per token (every token, or those of `list` in grid-stride order).
// Expert e lives in lane e % 32, slot e / 32.
__global__ void __launch_bounds__(kSelWarps * 32)
select_experts_kernel(const float* __restrict__ logits, const float* __restrict__ select_bias,
                      int32_t* __restrict__ topk_ids, float* __restrict__ topk_w, RouteParams rp, GateAudit au,
                      const int32_t* __restrict__ list, const int32_t* __restrict__ n_list) {
    pdl_enter();
    __shared__ float s_key[kSelWarps][kMaxE];
    __shared__ float s_sig[kSelWarps][kMaxE];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int n_tok = list ? *n_list : rp.T;
    for (int i = blockIdx.x * kSelWarps + warp; i < n_tok; i += gridDim.x * kSelWarps) {
    const int t = list ? list[i] : i;
    const int E = rp.E, k = rp.top_k;
    const float* l = logits + (size_t)t * E;
    float* key = s_key[warp];
    float* sig = s_sig[warp];
    const bool sigmoid = rp.score == GBMOE_SIGMOID;
    const int G = sigmoid ? rp.n_group : 1;
    const int gs = E / G;
    int sel_id = 0;
    float top_key = 0.0f;
    {
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

        // groups kept (bit g set); all experts allowed without group limiting.
        // margin_g: gap between the last kept and the best dropped group score
        uint32_t kept = 0xffffffffu;
        float margin_g = INFINITY;
        if (G > 1) {
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
            float last = 0.0f;
            for (int r = 0; r <= rp.topk_group && r < G; ++r) {
                float kk = (lane < G && !taken) ? gscore : -INFINITY;
                int ii = (lane < G && !taken) ? lane : kNone;
                warp_best(kk, ii);
                if (r == rp.topk_group) {  // the best dropped group
                    margin_g = last - kk;
                    break;
                }
                if (ii < 32) kept |= 1u << ii;  // always: topk_group <= G groups hold candidates
                if (lane == ii) taken = true;
                last = kk;
            }
        }

        // top-k over allowed experts, descending key, ties to the lower index;
        // margin_k: smallest gap between consecutive keys of the k chosen and
        // the best one left out
        uint32_t used = 0u;  // bit s: expert lane + 32 s already chosen
        float prev = 0.0f, margin_k = INFINITY;
        for (int j = 0; j <= k; ++j) {
            float kk = -INFINITY;
            int ii = kNone;
            for (int s = 0, e = lane; e < E; ++s, e += 32) {
                if ((used >> s) & 1u) continue;
                if (!((kept >> (e / gs)) & 1u)) continue;
                float v = key[e];
                if (ii == kNone || better(v, e, kk, ii)) { kk = v; ii = e; }
            }
            warp_best(kk, ii);
            if (j > 0 && ii < E) margin_k = fminf(margin_k, prev - kk);
            if (j == k) break;  // only the margin to the best expert left out
            // ii < E always (check_config keeps top_k within the kept groups' experts)
            if (ii < E && (ii & 31) == lane) used |= 1u << (ii >> 5);
            if (j == 0) top_key = kk;
            if (lane == j) sel_id = ii < E ? ii : 0;
            prev = kk;
        }

        if (au.x) {
        // bound on the logit error, and on the key error it causes (sigmoid:
        // slope <= 1/4, plus a few units in the last place of the fp32 key)
        float xx = 0.0f;
        const __nv_bfloat16* xt = au.x + (size_t)t * rp.H;
        for (int c = lane; c < rp.H / 8; c += 32) {
            float xv[8];
            Vec8<__nv_bfloat16>::load(xt + 8 * c, xv);
#pragma unroll
            for (int i = 0; i < 8; ++i) xx = fmaf(xv[i], xv[i], xx);
        }
#pragma unroll
        for (int d = 16; d >= 1; d >>= 1) xx += __shfl_xor_sync(0xffffffffu, xx, d);
        // (plus a few units in the last place of the logits, for the bias add)
        const float bl = au.scale * sqrtf(xx) * *au.wnorm_max + 1e-6f * (1.0f + fabsf(top_key));
        const float bk = sigmoid ? 0.25f * bl + 1e-6f : bl;
        const bool close = !(margin_k > 2.0f * bk) || !(margin_g > 4.0f * bk);
        if (close && lane == 0) au.flagged[atomicAdd(au.n_flagged, 1)] = t;
        }
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
    __syncwarp();
    }
}

// max over experts of ||wg[e]||_2 (fp32) into *out (zeroed beforehand): a
// warp per router row; the maximum taken on the float bits, which order like
// the values for non-negative floats
__global__ void __launch_bounds__(256)
row_norm_max_kernel(const __nv_bfloat16* __restrict__ wg, int E, int H, float* __restrict__ out) {
    pdl_enter();
    const int lane = threadIdx.x & 31;
    const int e = blockIdx.x * 8 + (threadIdx.x >> 5);
    if (e >= E) return;
    float ss = 0.0f;
    for (int c = lane; c < H / 8; c += 32) {
        float v[8];
        Vec8<__nv_bfloat16>::load(wg + (size_t)e * H + 8 * c, v);
#pragma unroll
        for (int i = 0; i < 8; ++i) ss = fmaf(v[i], v[i], ss);
    }
#pragma unroll
    for (int d = 16; d >= 1; d >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, d);
    if (lane == 0) atomicMax(reinterpret_cast<int*>(out), __float_as_int(sqrtf(ss)));
}

// Bound on |tensor-core logit - fixed-order logit| / (||x_t|| * max_e ||w_e||)
// that the audit uses (from measured differences on the workloads, with a
// safety factor; GBMOE_GATE_AUDIT_SCALE overrides it for tests).
constexpr float kGateAuditScale = 2.0e-6f;

static float gate_audit_scale() {
    const char* v = std::getenv("GBMOE_GATE_AUDIT_SCALE");
    if (!v || !*v) return kGateAuditScale;
    char* end = nullptr;
    const float f = std::strtof(v, &end);
    return (end != v && *end == '\0' && f >= 0.0f) ? f : kGateAuditScale;
}

// shared-memory size of the tiled gate kernel, set once per device
static cudaError_t gate_tiled_smem() {
    static DeviceOnce smem_set;
    return smem_set.run([] {
        return cudaFuncSetAttribute(gate_logits_tiled_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    (int)kGateTiledSmem);
    });
}

// ------------------------------------------------ RMSNorm before the gate

// y = x / sqrt(mean(x^2) + eps) * gamma per row, in the order of the gate's
// logits (its output decides the routing): one warp per row; lane l takes
// the 8-element chunks l, l+32, ... and sums their squares with one fused
// multiply-add each; the 32 partial sums are combined by the butterfly of
// pairwise additions; then ms = ss / H, v = ms + eps, r = sqrt(v), inv = 1 / r
// and y = (x * inv) * gamma, every step one correctly rounded fp32
// operation; y is rounded once to the activation type.
template <typename TA>
__global__ void __launch_bounds__(256)
rmsnorm_kernel(const TA* __restrict__ x, const TA* __restrict__ gamma, float eps, int T, int H, TA* __restrict__ y) {
    pdl_enter();
    const int lane = threadIdx.x & 31;
    const int64_t t = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
    if (t >= T) return;
    const TA* xr = x + t * H;
    float ss = 0.0f;
    for (int c = lane; c < H / 8; c += 32) {
        float v[8];
        Vec8<TA>::load(xr + 8 * c, v);
#pragma unroll
        for (int i = 0; i < 8; ++i) ss = __fmaf_rn(v[i], v[i], ss);
    }
#pragma unroll
    for (int d = 16; d >= 1; d >>= 1) ss = __fadd_rn(ss, __shfl_xor_sync(0xffffffffu, ss, d));
    const float ms = __fdiv_rn(ss, (float)H);
    const float inv = __fdiv_rn(1.0f, __fsqrt_rn(__fadd_rn(ms, eps)));
    for (int c = lane; c < H / 8; c += 32) {
        float v[8], g[8], o[8];
        Vec8<TA>::load(xr + 8 * c, v);
        Vec8<TA>::load(gamma + 8 * c, g);
#pragma unroll
        for (int i = 0; i < 8; ++i) o[i] = __fmul_rn(__fmul_rn(v[i], inv), g[i]);
        Vec8<TA>::store(y + t * H + 8 * c, o);
    }
}

cudaError_t launch_rmsnorm(const void* x, const void* gamma, float eps, int T, int H, int act_dtype, void* y,
                           cudaStream_t stream) {
    if (T == 0) return cudaSuccess;
    const dim3 grid((unsigned)((T + 7) / 8));
    cudaError_t le;
    if (act_dtype == GBMOE_BF16)
        le = launch_k(rmsnorm_kernel<__nv_bfloat16>, grid, dim3(256), 0, stream, static_cast<const __nv_bfloat16*>(x),
                      static_cast<const __nv_bfloat16*>(gamma), eps, T, H, static_cast<__nv_bfloat16*>(y));
    else
        le = launch_k(rmsnorm_kernel<float>, grid, dim3(256), 0, stream, static_cast<const float*>(x),
                      static_cast<const float*>(gamma), eps, T, H, static_cast<float*>(y));
    if (le != cudaSuccess) return le;
    return cudaGetLastError();
}

cudaError_t launch_route(const RouteParams& rp, const void* x, const void* wg, const float* logit_bias,
                         const float* select_bias, float* logits, int32_t* topk_ids, float* topk_w,
                         const RouteScratch& rs, cudaStream_t stream) {
    if (rp.T == 0) return cudaSuccess;
    const int ey = (rp.E + kGateWarps * kGateExpertsPerWarp - 1) / (kGateWarps * kGateExpertsPerWarp);
    dim3 block(kGateWarps * 32);
    GateAudit au{};
    if (rp.gate_tc) {
        // tensor-core logits, then the audited choice
        auto xp = static_cast<const __nv_bfloat16*>(x);
        auto wp = static_cast<const __nv_bfloat16*>(wg);
        if (const cudaError_t me = cudaMemsetAsync(rs.audit, 0, 8, stream); me != cudaSuccess)  // norm max, count
            return me;
        if (const cudaError_t le = launch_k(row_norm_max_kernel, dim3((rp.E + 7) / 8), dim3(256), 0, stream, wp,
                rp.E, rp.H, rs.audit); le != cudaSuccess)
            return le;
        if (const cudaError_t le = launch_gate_tc(x, wg, logit_bias, logits, rp.T, rp.H, rp.E, rs.sched, rs.err,
                stream); le != cudaSuccess)
            return le;
        au.x = xp; au.wnorm_max = rs.audit; au.scale = gate_audit_scale();
        au.flagged = rs.flagged; au.n_flagged = reinterpret_cast<int32_t*>(rs.audit + 1);
    } else if (rp.act_dtype == GBMOE_BF16) {
        auto xp = static_cast<const __nv_bfloat16*>(x);
        auto wp = static_cast<const __nv_bfloat16*>(wg);
        if (rp.T >= 1024) {
            if (const cudaError_t e = gate_tiled_smem(); e != cudaSuccess) return e;
            dim3 grid((rp.T + kGT - 1) / kGT, (rp.E + kGE - 1) / kGE);
            if (const cudaError_t le = launch_k(gate_logits_tiled_kernel, dim3(grid), dim3(256), kGateTiledSmem,
                    stream, xp, wp, logit_bias, logits, rp.T, rp.H, rp.E, static_cast<const int32_t*>(nullptr),
                    static_cast<const int32_t*>(nullptr)); le != cudaSuccess)
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
            dim3(kSelWarps * 32), 0, stream, logits, select_bias, topk_ids, topk_w, rp, au,
            static_cast<const int32_t*>(nullptr), static_cast<const int32_t*>(nullptr)); le != cudaSuccess)
        return le;
    if ((err = cudaGetLastError()) != cudaSuccess || !rp.gate_tc) return err;
    // flagged tokens: fixed-order logits, then their choice again (no audit)
    const int32_t* n_flag = reinterpret_cast<const int32_t*>(rs.audit + 1);
    if ((err = gate_tiled_smem()) != cudaSuccess) return err;
    const dim3 lgrid((rp.T + kGT - 1) / kGT, (rp.E + kGE - 1) / kGE);  // tiles past the flagged count exit
    if (const cudaError_t le = launch_k(gate_logits_tiled_kernel, lgrid, dim3(256), kGateTiledSmem, stream,
            static_cast<const __nv_bfloat16*>(x), static_cast<const __nv_bfloat16*>(wg), logit_bias, logits, rp.T,
            rp.H, rp.E, static_cast<const int32_t*>(rs.flagged), n_flag); le != cudaSuccess)
        return le;
    if ((err = cudaGetLastError()) != cudaSuccess) return err;
    const int blocks = sm_count() * 4;
    GateAudit none{};
    if (const cudaError_t le = launch_k(select_experts_kernel, dim3(blocks), dim3(kSelWarps * 32), 0, stream, logits,
            select_bias, topk_ids, topk_w, rp, none, static_cast<const int32_t*>(rs.flagged), n_flag);
        le != cudaSuccess)
        return le;
    return cudaGetLastError();
}

}  // namespace gbmoe
