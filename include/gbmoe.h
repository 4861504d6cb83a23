/*
 * gbmoe.h - C ABI of the GB300 (sm_103a) MoE layer forward.
 *
 * The layer is the paper's three-node MoE skeleton (Fig. 1, Section 1;
 * Fig. 3 and its discussion, Section 5.1):
 *   MoE Gate    router logits, top-k expert choice and routing weights
 *               -> moe_route
 *   Fused MoE   grouping of (token, slot) pairs by expert, then each expert's
 *               SwiGLU FFN on its rows, with bf16, fp8 (block-scaled E4M3,
 *               the format named in Section 6.2) or int4 weights
 *               -> moe_permute, moe_grouped_ffn, moe_shared_ffn
 *   Weight Sum  routing-weighted sum of each token's expert outputs
 *               -> moe_combine
 *   the whole layer -> moe_forward (device buffers) and moe_forward_hostio
 *   (host activations in and out).
 * The paper prints no formula for these nodes; the definitions stated below
 * are the standard ones, and the library reproduces an independent CPU
 * oracle of them (routing bit for bit, outputs within a per-dtype tolerance).
 *
 * Conventions for every call
 *  - Pointers are DEVICE pointers owned by the caller unless a parameter says
 *    host. Every tensor is dense, row-major, 16-byte aligned. The library
 *    never allocates, frees or synchronises (moe_device_status excepted);
 *    calls are asynchronous on `stream` (a cudaStream_t; NULL = the legacy
 *    default stream) and run on the current device.
 *  - Argument errors are found on the host before anything is launched and
 *    return a negative status; nothing is written then.
 *  - Calls that take a workspace use it for scratch only; its size comes from
 *    gbmoe_workspace_size for the same config. Calls sharing one workspace
 *    must not overlap in time (same stream, or ordered by events).
 *  - The library keeps per-device state for the life of the process (kernel
 *    shared-memory limits set once, SM counts, occupancy, the static
 *    scratch of moe_permute_noalloc). A reset of a device's context
 *    (cudaDeviceReset) discards what the driver held of it: make no further
 *    call on that device in the same process.
 *  - Names: T tokens, H hidden size, E routed experts, k = top_k, I expert
 *    intermediate size, P = T*k (token, slot) pairs, pair p = t*k + j.
 */
#ifndef GBMOE_H
#define GBMOE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Status codes. */
enum {
    GBMOE_OK = 0,
    GBMOE_EINVAL = -1,          /* null/misaligned pointer, inconsistent config */
    GBMOE_EUNSUPPORTED = -2,    /* valid config outside what the kernels cover  */
    GBMOE_EWORKSPACE = -3,      /* workspace smaller than gbmoe_workspace_size  */
    GBMOE_ECUDA = -4,           /* a CUDA launch or copy failed                 */
    GBMOE_EDEVICE_TIMEOUT = -5  /* a bounded device-side wait gave up           */
};

/* Element types. act_dtype uses F32 or BF16; w_dtype any of the five. */
enum {
    GBMOE_F32 = 0,
    GBMOE_BF16 = 1,
    GBMOE_FP8_E4M3_B128 = 2, /* e4m3 codes + fp32 scale per 128x128 block      */
    GBMOE_INT4_G128 = 3,     /* packed int4 + bf16 scale per 128 along K (row) */
    GBMOE_MXFP4 = 4          /* packed FP4 E2M1 + E8M0 scale per 32 along K    */
};

/* Router scoring. */
enum { GBMOE_SOFTMAX = 0, GBMOE_SIGMOID = 1 };

/* Which expert-FFN kernels run. GBMOE_FFN_TC_FP8 (FP8_E4M3_B128 weights and
 * bf16 activations only) multiplies the stored e4m3 weights on the fp8 tensor
 * cores: each GEMM's input rows (x, then h) are brought to e4m3 with one fp32
 * scale s per row and 128 consecutive k (s = amax / 448) as two codes,
 * q1 = e4m3(x / s) and q2 = e4m3(x / s - q1), so that x = s * (q1 + q2) to
 * within max(2^-8 |x / s|, 2^-10) * s, a bf16-like precision; both codes are
 * multiplied with the weights and each 128-wide k block's partial sum is
 * scaled by both blocks' scales and accumulated in fp32. AUTO takes it for
 * fp8 weights whenever a tensor-core route applies.
 * AUTO streams weights when the average number
 * of rows per expert P/E is at most 16 and otherwise runs the grouped GEMM
 * (tensor cores for bf16 activations, CUDA cores for fp32). On the tensor
 * cores, int4/MXFP4 weights are decoded inside the GEMM when P/E < 256; with
 * more rows per expert (several M tiles reuse each weight tile) AUTO takes
 * GBMOE_FFN_TC_DEQUANT: one pass decodes the active experts' weights to a
 * bf16 copy in the workspace (the same bf16 values the in-GEMM decode makes),
 * then the bf16 GEMM runs on it. The _PAIR routes run the same GEMM on CTA
 * pairs (tcgen05 cta_group::2): one MMA of 256 rows per pair, each CTA
 * holding 128 rows of A and half of the bf16 weight tile, which halves the
 * weight bytes each SM reads per MMA; an expert's rows are then covered in
 * 256-row tiles, so AUTO takes them only from P/E >= 1024 (little padding).
 * Their outputs equal the one-CTA routes' bit for bit. TC_PAIR needs bf16
 * weights; quantised weights take TC_PAIR_DEQUANT. */
enum {
    GBMOE_FFN_AUTO = 0,
    GBMOE_FFN_STREAM = 1,     /* weight streaming: few rows per expert (decode)       */
    GBMOE_FFN_SIMT = 2,       /* CUDA-core tiled GEMM (fp32 activations, any weights) */
    GBMOE_FFN_TC = 3,         /* tcgen05/TMEM/TMA grouped GEMM (bf16 activations)     */
    GBMOE_FFN_TC_DEQUANT = 4, /* as TC, quantised weights decoded once beforehand     */
    GBMOE_FFN_TC_FP8 = 5,     /* fp8 tensor cores: FP8_E4M3_B128 weights as stored,
                                 activations quantised to e4m3 per 1x128 block      */
    GBMOE_FFN_TC_PAIR = 6,    /* as TC on CTA pairs: one MMA of 256 rows per pair
                                 (each CTA holds half the weight tile); bf16
                                 weights only (quantised: TC_PAIR_DEQUANT)          */
    GBMOE_FFN_TC_PAIR_DEQUANT = 7 /* as TC_DEQUANT, the bf16 GEMM on CTA pairs      */
};

/* How the MoE Gate computes the router logits. SIMT: CUDA cores in the fixed
 * order of the definition (moe_route). TC: tensor cores (bf16 activations
 * only), whose fp32 sums run in the hardware's order; each token's expert
 * choice is then audited: when any comparison that decides it (the order of
 * the chosen keys, the chosen against the best one left out, and the last
 * kept group against the best dropped one) is closer than a bound on the
 * difference between the two orders (scale * ||x_t|| * max_e ||w_e||, plus a
 * few units in the last place), that token's logits are recomputed in the
 * fixed order and its choice is made again, so the ids equal the SIMT
 * route's. The scale (2e-6) is four times the largest difference measured on
 * the benchmark workloads, not a worst-case bound. The routing weights of
 * tokens not recomputed come from the tensor-core logits: within about 1e-4
 * relative of the SIMT route's. AUTO: TC for bf16 batches of 256 tokens or
 * more, else SIMT. */
enum { GBMOE_GATE_AUTO = 0, GBMOE_GATE_SIMT = 1, GBMOE_GATE_TC = 2 };

/* Where moe_forward computes the Weight Sum. SEPARATE: moe_combine's gather
 * kernel after the FFN. FUSED (tensor-core FFN routes GBMOE_FFN_TC,
 * _TC_DEQUANT, _TC_PAIR and _TC_PAIR_DEQUANT): in the down GEMM's epilogue, which writes topk_w * y of each
 * pair into a slot buffer in pair order and counts, per token and 256 output
 * columns, the slots written; the warp that writes the last one sums the
 * token's slots in slot order (plus the shared expert's row, computed before
 * the routed FFN) and writes out once: deterministic, no atomics on data.
 * The slot is rounded to bf16 after the weight multiply (SEPARATE multiplies
 * the bf16 row), so the two differ within rounding. Other FFN routes use
 * SEPARATE. AUTO: SEPARATE (measured faster on GB300). */
enum { GBMOE_COMBINE_AUTO = 0, GBMOE_COMBINE_SEPARATE = 1, GBMOE_COMBINE_FUSED = 2 };

typedef struct gbmoe_config {
    int32_t T, H, I, E, top_k;
    int32_t score;        /* GBMOE_SOFTMAX or GBMOE_SIGMOID                         */
    int32_t renormalize;  /* 1: the selected experts' weights sum to routed_scale   */
    int32_t n_group;      /* sigmoid only: E experts in n_group contiguous groups   */
    int32_t topk_group;   /* sigmoid only: groups kept before the expert choice     */
    float routed_scale;   /* multiplies every routing weight (1.0 = none)           */
    int32_t act_dtype;    /* x, router weight, intermediates, out: F32 or BF16      */
    int32_t w_dtype;      /* routed and shared expert weights                       */
    int32_t has_shared;   /* 1: add one always-on expert with weight 1              */
    int32_t I_shared;     /* its intermediate size                                  */
    int32_t ffn_route;    /* GBMOE_FFN_*                                            */
    int32_t gate_route;   /* GBMOE_GATE_*                                           */
    int32_t combine_route; /* GBMOE_COMBINE_*                                       */
} gbmoe_config;

/* One set of expert weights (all experts stacked, E of them, or 1 for the
 * shared expert). nn.Linear layout: gate and up are [E, I, H], down is
 * [E, H, I] (output rows, input contiguous).
 *  F32 / BF16:      w_* hold the values; s_* are NULL.
 *  FP8_E4M3_B128:   w_* hold e4m3 bytes in the same shape; s_gate, s_up are
 *                   fp32 [E, I/128, H/128] and s_down fp32 [E, H/128, I/128];
 *                   W[n,k] = e4m3(q[n,k]) * s[n/128][k/128].
 *  INT4_G128:       w_* hold packed nibbles, [E, N, K/2] bytes for an [N, K]
 *                   matrix, element 2i in the low nibble of byte i, two's
 *                   complement; s_* are bf16 [E, N, K/128];
 *                   W[n,k] = q[n,k] * s[n][k/128].
 *  MXFP4:           the OCP Microscaling FP4 format, the MXFP4 expert weights
 *                   of the DeepSeek reference path (Section 6.2): w_* hold
 *                   packed FP4 E2M1 nibbles laid out as for INT4_G128 (sign in
 *                   bit 3, 2 exponent bits with bias 1, 1 mantissa bit:
 *                   0, 0.5, 1, 1.5, 2, 3, 4, 6); s_* are E8M0 bytes
 *                   [E, N, K/32], 2-byte aligned;
 *                   W[n,k] = e2m1(q[n,k]) * 2^(s[n][k/32] - 127). Decoding
 *                   to bf16 or fp32 is exact. */
typedef struct gbmoe_expert_weights {
    const void *w_gate, *w_up, *w_down;
    const void *s_gate, *s_up, *s_down;
} gbmoe_expert_weights;

/* Human-readable name of a status code (static string). */
const char* gbmoe_status_string(int status);

/* The CUDA runtime error code (a cudaError_t value) behind the last
 * GBMOE_ECUDA this thread received from the library, or 0 if none; the
 * library links its own copy of the CUDA runtime, so the caller's
 * cudaGetLastError does not see it. Cleared by reading. */
int gbmoe_last_cuda_error(void);

/* GBMOE_OK if the config is valid and covered, else the status a call with it
 * would return. Limits: H % 256 == 0, I % 128 == 0 (I_shared too),
 * 1 <= E <= 512, 1 <= top_k <= min(E, 32), T >= 0, P <= 2^30; with fp8
 * weights also P * kb < 2^31 and E * kb^2 < 2^31, kb = max(H, I, I_shared) /
 * 128 (the fp8 route indexes its scale tensors with 32-bit offsets). */
int gbmoe_check_config(const gbmoe_config* cfg);

/* Workspace bytes that moe_forward / moe_forward_hostio need for cfg (the
 * other calls need no more). 0 if the config is invalid. */
size_t gbmoe_workspace_size(const gbmoe_config* cfg);

/* The FFN route (one of GBMOE_FFN_STREAM .. _TC_PAIR_DEQUANT) that moe_forward runs for
 * cfg: for the routed experts (shared = 0) or the shared expert (shared = 1).
 * Negative status if the config is invalid. */
int gbmoe_ffn_route(const gbmoe_config* cfg, int shared);

/* The gate route (GBMOE_GATE_SIMT or _TC) that moe_route and moe_forward run
 * for cfg. Negative status if the config is invalid. */
int gbmoe_gate_route(const gbmoe_config* cfg);

/*
 * RMSNorm of the layer input, the step before the MoE Gate: for every row t,
 *   y[t,:] = x[t,:] / sqrt(mean(x[t,:]^2) + eps) * gamma,
 * in fp32 in the gate's fixed order (sum of squares: 32 partial sums over
 * the 8-element chunks p, p+32, ... with one fused multiply-add per element,
 * then the pairwise sums for d = 16..1; then mean, + eps, sqrt, reciprocal
 * and the two products, each one correctly rounded fp32 operation), rounded
 * once to act_dtype. Its output is the x that moe_route / moe_forward take:
 * the experts' choice follows from it bit for bit. x, y [T, H] and gamma [H]
 * are act_dtype device pointers (16-byte aligned; y may not overlap x);
 * eps >= 0 and finite. Uses cfg's T, H and act_dtype only. No workspace.
 */
int moe_rmsnorm(const gbmoe_config* cfg, const void* x, const void* gamma, float eps, void* y, void* stream);

/*
 * MoE Gate (Fig. 1 and Fig. 3). For every token t:
 *   l[t,e] = x[t,:] . w_router[e,:] (+ logit_bias[e]), fp32, in a fixed order:
 *     32 partial sums, partial p takes the 8-element chunks p, p+32, ... in
 *     order with one fused multiply-add per element, then pairwise sums
 *     s[p] + s[p xor d] for d = 16, 8, 4, 2, 1, then one fp32 add of the bias;
 *   softmax: top_k largest l (ties to the lower expert) in descending order;
 *     weight = exp(l_j - max) / sum over the selected (renormalize) or over
 *     all E (otherwise), times routed_scale;
 *   sigmoid: s_e = 1/(1 + exp(-l_e)) with a fixed fp32 exponential,
 *     q_e = s_e + select_bias[e]; keep the topk_group groups whose two
 *     largest q sum highest (ties to the lower group), then the top_k largest
 *     q in kept groups (ties to the lower expert); weight = s_j / sum of
 *     selected s (renormalize) or s_j, times routed_scale.
 * x [T, H] and w_router [E, H] are act_dtype. logit_bias [E] fp32 or NULL
 * (enters the logit, so weights too); select_bias [E] fp32 or NULL (sigmoid
 * selection only). Writes topk_ids [T, k] int32 and topk_w [T, k] fp32.
 * Workspace: the logits (T*E fp32).
 */
int moe_route(const gbmoe_config* cfg, const void* x, const void* w_router, const float* logit_bias,
              const float* select_bias, int32_t* topk_ids, float* topk_w, void* workspace,
              size_t workspace_bytes, void* stream);

/*
 * Fused MoE, grouping step: stable counting sort of the P pairs by expert.
 * topk_ids [T, k] int32, each in [0, E). Writes counts [E], offsets [E+1]
 * (exclusive prefix sum, offsets[E] = P), sorted_pair [P] (pairs ordered by
 * expert, then by pair index) and pair_pos [P] (inverse: position of pair p),
 * all int32. Bit-exact and deterministic. A pair whose id is out of range is
 * dropped: it is not counted and gets no slot; its pair_pos entry is -1,
 * offsets[E] is then below P, and sorted_pair[offsets[E] .. P-1] hold -1.
 * moe_grouped_ffn and moe_combine accept these outputs as they are: the FFN
 * computes only the counted rows, and a dropped pair adds nothing to its
 * token's output.
 */
int moe_permute(const gbmoe_config* cfg, const int32_t* topk_ids, int32_t* counts, int32_t* offsets,
                int32_t* sorted_pair, int32_t* pair_pos, void* workspace, size_t workspace_bytes,
                void* stream);

/*
 * Fused MoE, expert FFNs. For every sorted position r of expert e
 * (offsets[e] <= r < offsets[e+1]) with token t = sorted_pair[r] / k:
 *   g = Wgate_e x_t, u = Wup_e x_t, a = silu(g) * u, y_pairs[r] = Wdown_e a.
 * fp32 accumulation; a (the intermediate) and y_pairs are stored in
 * act_dtype. No routing weight is applied here. x [T, H] act_dtype; counts,
 * offsets, sorted_pair as produced by moe_permute; y_pairs [P, H] act_dtype.
 */
int moe_grouped_ffn(const gbmoe_config* cfg, const void* x, const int32_t* counts, const int32_t* offsets,
                    const int32_t* sorted_pair, const gbmoe_expert_weights* experts, void* y_pairs,
                    void* workspace, size_t workspace_bytes, void* stream);

/*
 * Shared expert: y_shared[t] = SwiGLU FFN of x_t with the single expert
 * `shared` (intermediate size I_shared, same w_dtype), for every token.
 * y_shared [T, H] act_dtype. Requires cfg->has_shared.
 */
int moe_shared_ffn(const gbmoe_config* cfg, const void* x, const gbmoe_expert_weights* shared,
                   void* y_shared, void* workspace, size_t workspace_bytes, void* stream);

/*
 * Weight Sum (Fig. 1 and Fig. 3):
 *   out[t] = sum_{j=0..k-1} topk_w[t,j] * y_pairs[pair_pos[t*k + j]]
 *            (+ y_shared[t] if y_shared is not NULL),
 * summed in fp32 in that order and rounded once to act_dtype. A gather per
 * token: no atomics, deterministic. Slots with a negative pair_pos (pairs
 * moe_permute dropped) are skipped. y_pairs [P, H], y_shared [T, H] or NULL,
 * out [T, H], all act_dtype; topk_w [T, k] fp32; pair_pos [P] int32.
 */
int moe_combine(const gbmoe_config* cfg, const void* y_pairs, const float* topk_w, const int32_t* pair_pos,
                const void* y_shared, void* out, void* stream);

/*
 * The whole layer: moe_route, moe_permute, moe_grouped_ffn, moe_shared_ffn
 * (if cfg->has_shared) and moe_combine in sequence on one stream, with all
 * intermediates in the workspace. out [T, H] act_dtype. Optional outputs
 * (NULL to skip): topk_ids [T, k] int32, topk_w [T, k] fp32, counts [E] int32.
 * shared may be NULL only when cfg->has_shared is 0.
 */
int moe_forward(const gbmoe_config* cfg, const void* x, const void* w_router, const float* logit_bias,
                const float* select_bias, const gbmoe_expert_weights* experts,
                const gbmoe_expert_weights* shared, void* out, int32_t* topk_ids, float* topk_w,
                int32_t* counts, void* workspace, size_t workspace_bytes, void* stream);

/*
 * moe_forward with HOST activations: copies x_host [T, H] to the device,
 * runs the layer, copies the result to out_host [T, H] (both act_dtype, on
 * `stream`, asynchronous: synchronise the stream before reading out_host;
 * use page-locked host memory for truly asynchronous copies). Weights and the
 * other arguments are device pointers as in moe_forward.
 */
int moe_forward_hostio(const gbmoe_config* cfg, const void* x_host, const void* w_router,
                       const float* logit_bias, const float* select_bias,
                       const gbmoe_expert_weights* experts, const gbmoe_expert_weights* shared,
                       void* out_host, void* workspace, size_t workspace_bytes, void* stream);

/*
 * Reads (and clears) the device error word that bounded device-side waits
 * set in `workspace`, after synchronising `stream`. *status receives GBMOE_OK
 * or GBMOE_EDEVICE_TIMEOUT. This is the only call that synchronises.
 * The waits are those of the tensor-core FFN kernels (the GBMOE_FFN_TC*
 * routes): each gives up after 2 s, stops issuing work, lets the copies
 * and MMAs it issued finish, and sets the word; the call's outputs are then
 * incomplete. For tests of this path the environment variable
 * GBMOE_TC_WAIT_LIMIT_NS (read at every call) lowers the limit, in ns.
 */
int moe_device_status(void* workspace, void* stream, int32_t* status);

/*
 * moe_permute without a workspace: the same grouping as moe_permute (same
 * outputs, bit for bit), with its scratch held in a static device array
 * inside this library instead of a caller buffer. The paper has no
 * counterpart; this exists for callers that cannot allocate device memory
 * for a call: plain C hosts with no device allocator of their own, serving
 * engines that reserve all device memory up front and lend out no scratch,
 * and code that runs where cudaMalloc is not allowed. The array is 1 MiB
 * (262144 int32) per device, held by every GPU that loads the library until
 * the process exits; problems needing more, 2 * ceil(T*k / 1024) * E ints,
 * return GBMOE_EUNSUPPORTED without launching anything. The call allocates
 * nothing. Its first call on each device looks up the array's device
 * address (cudaGetSymbolAddress, with that device current), so make that
 * first call before any stream capture. The looked-up address is kept for
 * the life of the process and does not survive a reset of the device's
 * context (cudaDeviceReset): do not call this after one. All calls share
 * the array: calls that overlap on the GPU (unordered streams) race; order
 * them.
 */
int moe_permute_noalloc(const gbmoe_config* cfg, const int32_t* topk_ids, int32_t* counts, int32_t* offsets,
                        int32_t* sorted_pair, int32_t* pair_pos, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* GBMOE_H */
