// C ABI of the MoE layer (declared in include/gbmoe.h): argument checks on
// the host, workspace carving, and the launch sequence of the layer's nodes
// (MoE Gate -> Fused MoE -> Weight Sum) on the caller's stream.
#include <algorithm>
#include <climits>
#include <cmath>
#include <cstdint>
#include <cstring>

#include "common.cuh"
#include "ffn_sched.h"
#include "kernels.h"

using namespace gbmoe;

namespace {

constexpr size_t kAlign = 256;

size_t align_up(size_t v) { return (v + kAlign - 1) & ~(kAlign - 1); }

size_t act_bytes(int act) { return act == GBMOE_F32 ? 4 : 2; }

bool quantised_weights(int w) { return w == GBMOE_FP8_E4M3_B128 || w == GBMOE_INT4_G128 || w == GBMOE_MXFP4; }
// routes that run the bf16-operand tensor-core GEMM (launch_ffn_tc)
bool bf16_gemm_route(int r) {
    return r == GBMOE_FFN_TC || r == GBMOE_FFN_TC_DEQUANT || r == GBMOE_FFN_TC_PAIR || r == GBMOE_FFN_TC_PAIR_DEQUANT;
}
bool pair_route(int r) { return r == GBMOE_FFN_TC_PAIR || r == GBMOE_FFN_TC_PAIR_DEQUANT; }
bool dequant_route(int r) { return r == GBMOE_FFN_TC_DEQUANT || r == GBMOE_FFN_TC_PAIR_DEQUANT; }

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

int check_cfg(const gbmoe_config* c) {
    if (!c) return GBMOE_EINVAL;
    if (c->T < 0 || c->H <= 0 || c->I <= 0 || c->E <= 0 || c->top_k <= 0) return GBMOE_EINVAL;
    if (c->top_k > c->E) return GBMOE_EINVAL;
    if (c->score != GBMOE_SOFTMAX && c->score != GBMOE_SIGMOID) return GBMOE_EINVAL;
    if (c->act_dtype != GBMOE_F32 && c->act_dtype != GBMOE_BF16) return GBMOE_EINVAL;
    if (c->w_dtype < GBMOE_F32 || c->w_dtype > GBMOE_MXFP4) return GBMOE_EINVAL;
    if (c->has_shared != 0 && c->has_shared != 1) return GBMOE_EINVAL;
    if (c->has_shared && c->I_shared <= 0) return GBMOE_EINVAL;
    if (c->ffn_route < GBMOE_FFN_AUTO || c->ffn_route > GBMOE_FFN_TC_PAIR_DEQUANT) return GBMOE_EINVAL;
    if (c->gate_route < GBMOE_GATE_AUTO || c->gate_route > GBMOE_GATE_TC) return GBMOE_EINVAL;
    if (c->gate_route == GBMOE_GATE_TC && c->act_dtype != GBMOE_BF16) return GBMOE_EUNSUPPORTED;
    if (c->combine_route < GBMOE_COMBINE_AUTO || c->combine_route > GBMOE_COMBINE_FUSED) return GBMOE_EINVAL;
    if (!std::isfinite(c->routed_scale)) return GBMOE_EINVAL;
    if (c->score == GBMOE_SIGMOID) {
        if (c->n_group < 1 || c->E % c->n_group != 0) return GBMOE_EINVAL;
        if (c->n_group > 1 && c->E / c->n_group < 2) return GBMOE_EINVAL;
        if (c->topk_group < 1 || c->topk_group > c->n_group) return GBMOE_EINVAL;
        if ((int64_t)c->top_k > (int64_t)c->topk_group * (c->E / c->n_group)) return GBMOE_EINVAL;
    }
    // what the kernels cover
    if (c->H % 256 != 0 || c->I % 128 != 0) return GBMOE_EUNSUPPORTED;
    if (c->has_shared && c->I_shared % 128 != 0) return GBMOE_EUNSUPPORTED;
    if (c->E > 512 || c->top_k > 32) return GBMOE_EUNSUPPORTED;
    if (c->score == GBMOE_SIGMOID && c->n_group > 32) return GBMOE_EUNSUPPORTED;
    if ((int64_t)c->T * c->top_k > (int64_t(1) << 30)) return GBMOE_EUNSUPPORTED;
    if (c->act_dtype == GBMOE_BF16 && c->w_dtype == GBMOE_F32) return GBMOE_EUNSUPPORTED;
    if (bf16_gemm_route(c->ffn_route) && c->act_dtype != GBMOE_BF16) return GBMOE_EUNSUPPORTED;
    if (c->ffn_route == GBMOE_FFN_TC_FP8 && (c->act_dtype != GBMOE_BF16 || c->w_dtype != GBMOE_FP8_E4M3_B128))
        return GBMOE_EUNSUPPORTED;
    if (c->w_dtype == GBMOE_FP8_E4M3_B128) {
        // the fp8 route addresses its activation and weight scales with 32-bit
        // offsets (far more rows than any device could hold the codes of)
        const int64_t kb = std::max({c->H, c->I, c->has_shared ? c->I_shared : 0}) / 128;
        if ((int64_t)c->T * c->top_k * kb > INT32_MAX || (int64_t)c->E * kb * kb > INT32_MAX)
            return GBMOE_EUNSUPPORTED;
    }
    return GBMOE_OK;
}

bool stream_fits(int act_dtype, int H, int I) { return stream_smem_bytes(act_dtype, H, I) <= stream_smem_budget(); }

// Kernel route for an FFN problem with n_rows rows over E experts.
int pick_route(const gbmoe_config* c, int64_t n_rows, int E, int I) {
    int r = c->ffn_route;
    if (r != GBMOE_FFN_AUTO) return r;
    if (n_rows <= 16 * (int64_t)E && stream_fits(c->act_dtype, c->H, I)) return GBMOE_FFN_STREAM;
    if (c->act_dtype == GBMOE_BF16) {
        FfnProblem probe{};
        probe.act_dtype = c->act_dtype;
        probe.w_dtype = c->w_dtype;
        probe.H = c->H;
        probe.I = I;
        probe.E = E;
        // fp8 weights: the fp8 tensor-core route (no decode; its two-term
        // activation codes keep bf16-level accuracy)
        if (ffn_tc_fp8_supported(probe)) return GBMOE_FFN_TC_FP8;
        if (ffn_tc_supported(probe)) {
            const bool dequant = quantised_weights(c->w_dtype) && n_rows >= kDequantRowsPerExpert * E;
            // CTA pairs (256-row tiles) once experts are deep enough that the
            // padding of their last tile stays small; they multiply bf16 tiles
            if (dequant) probe.w_dq = &probe;
            const bool pairs = n_rows >= kPairRowsPerExpert * E && ffn_tc_pair_supported(probe);
            if (dequant) return pairs ? GBMOE_FFN_TC_PAIR_DEQUANT : GBMOE_FFN_TC_DEQUANT;
            return pairs && c->w_dtype == GBMOE_BF16 ? GBMOE_FFN_TC_PAIR : GBMOE_FFN_TC;
        }
    }
    return GBMOE_FFN_SIMT;
}

// Bytes of the bf16 weight copy the TC_DEQUANT route decodes into (0 when
// the route of that problem does not use one).
size_t dequant_bytes(const gbmoe_config* c, int64_t n_rows, int E, int I) {
    if (!quantised_weights(c->w_dtype) || !dequant_route(pick_route(c, n_rows, E, I))) return 0;
    return (size_t)3 * E * c->H * I * 2;
}

// Bytes of the sorted copy of x the routed problem's GEMM reads (0 when its
// route does not read one: the one-CTA bf16 GEMM gathers its rows from x,
// the other routes read x or the fp8 codes directly).
size_t sorted_x_bytes(const gbmoe_config* c) {
    const int64_t P = (int64_t)c->T * c->top_k;
    const int r = pick_route(c, P, c->E, c->I);
    const bool reads_copy = pair_route(r) || (r == GBMOE_FFN_TC && quantised_weights(c->w_dtype));
    return reads_copy ? (size_t)P * c->H * act_bytes(c->act_dtype) : 0;
}

struct Layout {
    size_t err, audit, flagged, arrive, logits, ids, w, counts, offsets, sorted, pos, perm, sched, h, xs, y, ysh, xin, xout, wdq,
        wdq_sh, aq, as, hq, hs, total;
};

// true when the routed or the shared FFN problem of c runs on the fp8 route
bool uses_fp8_route(const gbmoe_config* c) {
    if (pick_route(c, (int64_t)c->T * c->top_k, c->E, c->I) == GBMOE_FFN_TC_FP8) return true;
    return c->has_shared && pick_route(c, c->T, 1, c->I_shared) == GBMOE_FFN_TC_FP8;
}

Layout layout(const gbmoe_config* c) {
    const int64_t T = c->T, P = (int64_t)c->T * c->top_k, E = c->E, H = c->H;
    const size_t ab = act_bytes(c->act_dtype);
    const int64_t rows_max = P > T ? P : T;
    const int64_t I_max = c->has_shared && c->I_shared > c->I ? c->I_shared : c->I;
    Layout L{};
    size_t o = 0;
    auto take = [&](size_t bytes) { size_t at = o; o = align_up(o + bytes); return at; };
    L.err = take(4);
    L.audit = take(8);
    L.flagged = take((size_t)T * 4);
    L.arrive = take((size_t)T * (H / 256) * 4);
    L.logits = take((size_t)T * E * 4);
    L.ids = take((size_t)P * 4);
    L.w = take((size_t)P * 4);
    L.counts = take((size_t)E * 4);
    L.offsets = take((size_t)(E + 1) * 4);
    L.sorted = take((size_t)P * 4);
    L.pos = take((size_t)P * 4);
    L.perm = take(permute_scratch_ints(P, (int)E) * 4);
    L.sched = take(ffn_sched_ints((int)(E > 1 ? E : 1), rows_max) * 4);
    L.h = take((size_t)rows_max * I_max * ab);
    L.xs = take(sorted_x_bytes(c));
    L.y = take((size_t)P * H * ab);
    L.ysh = take(c->has_shared ? (size_t)T * H * ab : 0);
    L.xin = take((size_t)T * H * ab);
    L.xout = take((size_t)T * H * ab);
    L.wdq = take(dequant_bytes(c, P, (int)E, c->I));
    L.wdq_sh = take(c->has_shared ? dequant_bytes(c, T, 1, c->I_shared) : 0);
    const bool f8 = uses_fp8_route(c);  // e4m3 copies of the GEMM inputs and their 1x128 scales
    L.aq = take(f8 ? (size_t)2 * rows_max * H : 0);  // two e4m3 code planes
    L.as = take(f8 ? (size_t)rows_max * (H / 128) * 4 : 0);
    L.hq = take(f8 ? (size_t)2 * rows_max * I_max : 0);
    L.hs = take(f8 ? (size_t)rows_max * (I_max / 128) * 4 : 0);
    L.total = o;
    return L;
}

template <typename T>
T* at(void* ws, size_t off) {
    return reinterpret_cast<T*>(static_cast<char*>(ws) + off);
}

thread_local int g_last_cuda_error = 0;  // gbmoe_last_cuda_error

int cuda_status(cudaError_t e) {
    if (e == cudaSuccess) return GBMOE_OK;
    g_last_cuda_error = (int)e;
    return GBMOE_ECUDA;
}

int check_ws(const gbmoe_config* c, void* ws, size_t bytes) {
    if (!ws || !aligned(ws, kAlign)) return GBMOE_EINVAL;
    if (bytes < layout(c).total) return GBMOE_EWORKSPACE;
    return GBMOE_OK;
}

int check_weights(const gbmoe_config* c, const gbmoe_expert_weights* w) {
    if (!w || !w->w_gate || !w->w_up || !w->w_down) return GBMOE_EINVAL;
    if (!aligned(w->w_gate, 16) || !aligned(w->w_up, 16) || !aligned(w->w_down, 16)) return GBMOE_EINVAL;
    if (quantised_weights(c->w_dtype)) {
        if (!w->s_gate || !w->s_up || !w->s_down) return GBMOE_EINVAL;
        const size_t sa = c->w_dtype == GBMOE_MXFP4 ? 2 : 4;  // E8M0 bytes are read in pairs
        if (!aligned(w->s_gate, sa) || !aligned(w->s_up, sa) || !aligned(w->s_down, sa)) return GBMOE_EINVAL;
    }
    return GBMOE_OK;
}

// Gate route: the fixed-order CUDA-core logits, or tensor-core logits audited
// against that order (AUTO: bf16 batches of at least kGateTcMinTokens tokens).
constexpr int kGateTcMinTokens = 256;

int pick_gate(const gbmoe_config* c) {
    if (c->gate_route != GBMOE_GATE_AUTO) return c->gate_route;
    if (c->act_dtype != GBMOE_BF16 || c->T < kGateTcMinTokens) return GBMOE_GATE_SIMT;
    FfnProblem probe{};
    probe.act_dtype = c->act_dtype;
    probe.w_dtype = GBMOE_BF16;
    probe.H = c->H;
    probe.I = 128;
    return ffn_tc_supported(probe) ? GBMOE_GATE_TC : GBMOE_GATE_SIMT;
}

RouteParams route_params(const gbmoe_config* c) {
    RouteParams rp;
    rp.T = c->T; rp.H = c->H; rp.E = c->E; rp.top_k = c->top_k;
    rp.score = c->score; rp.renormalize = c->renormalize; rp.n_group = c->n_group;
    rp.topk_group = c->topk_group; rp.routed_scale = c->routed_scale; rp.act_dtype = c->act_dtype;
    rp.gate_tc = pick_gate(c) == GBMOE_GATE_TC;
    return rp;
}

RouteScratch route_scratch(const gbmoe_config* c, void* ws) {
    const Layout L = layout(c);
    return RouteScratch{at<int32_t>(ws, L.sched), at<int32_t>(ws, L.err), at<float>(ws, L.audit),
                        at<int32_t>(ws, L.flagged)};
}

// GBMOE_OK when an FFN problem of intermediate size I can run on `route`,
// checked on the host so that a call fails before it enqueues anything.
int route_launchable(const gbmoe_config* c, int route, int I) {
    switch (route) {
        case GBMOE_FFN_STREAM: return stream_fits(c->act_dtype, c->H, I) ? GBMOE_OK : GBMOE_EUNSUPPORTED;
        case GBMOE_FFN_SIMT: return GBMOE_OK;
        case GBMOE_FFN_TC:
        case GBMOE_FFN_TC_DEQUANT:
        case GBMOE_FFN_TC_FP8:
        case GBMOE_FFN_TC_PAIR:
        case GBMOE_FFN_TC_PAIR_DEQUANT: {
            FfnProblem probe{};
            probe.act_dtype = c->act_dtype;
            probe.w_dtype = c->w_dtype;
            probe.H = c->H;
            probe.I = I;
            // the decode-once routes run the bf16 kernel (a non-null w_dq says so)
            if (route == GBMOE_FFN_TC_PAIR_DEQUANT && quantised_weights(c->w_dtype)) probe.w_dq = &probe;
            const bool ok = route == GBMOE_FFN_TC_FP8   ? ffn_tc_fp8_supported(probe)
                            : pair_route(route) ? ffn_tc_pair_supported(probe)
                                                : ffn_tc_supported(probe);
            return ok ? GBMOE_OK : GBMOE_EUNSUPPORTED;
        }
        default: return GBMOE_EINVAL;
    }
}

int run_ffn(const gbmoe_config* c, FfnProblem& p, int route, cudaStream_t stream) {
    if (int s = route_launchable(c, route, p.I)) return s;
    cudaError_t err;
    switch (route) {
        case GBMOE_FFN_STREAM: err = launch_ffn_stream(p, stream); break;
        case GBMOE_FFN_SIMT: err = launch_ffn_simt(p, stream); break;
        case GBMOE_FFN_TC_FP8: err = launch_ffn_tc_fp8(p, stream); break;
        default:  // GBMOE_FFN_TC, _TC_DEQUANT, _TC_PAIR, _TC_PAIR_DEQUANT
            p.cta_pair = pair_route(route) ? 1 : 0;
            err = launch_ffn_tc(p, stream);
            break;
    }
    return cuda_status(err);
}

// the fp8 route's scratch (the routed and the shared problem run one after
// the other, so they share it)
void set_fp8_buffers(FfnProblem& p, const Layout& L, void* ws) {
    p.a_q = at<char>(ws, L.aq);
    p.a_s = at<float>(ws, L.as);
    p.h_q = at<char>(ws, L.hq);
    p.h_s = at<float>(ws, L.hs);
}

FfnProblem routed_problem(const gbmoe_config* c, const void* x, const int32_t* counts, const int32_t* offsets,
                          const int32_t* sorted_pair, const gbmoe_expert_weights* w, void* y, void* ws) {
    const Layout L = layout(c);
    FfnProblem p{};
    p.x = x; p.counts = counts; p.offsets = offsets; p.sorted_pair = sorted_pair; p.pair_div = c->top_k;
    p.E = c->E; p.H = c->H; p.I = c->I; p.n_rows = (int64_t)c->T * c->top_k;
    p.act_dtype = c->act_dtype; p.w_dtype = c->w_dtype;
    p.w_gate = w->w_gate; p.w_up = w->w_up; p.w_down = w->w_down;
    p.s_gate = w->s_gate; p.s_up = w->s_up; p.s_down = w->s_down;
    p.y = y;
    p.h = at<char>(ws, L.h); p.sched = at<int32_t>(ws, L.sched);
    p.x_sorted = sorted_x_bytes(c) ? at<char>(ws, L.xs) : nullptr;
    p.err = at<int32_t>(ws, L.err);
    p.w_dq = dequant_bytes(c, p.n_rows, p.E, p.I) ? at<char>(ws, L.wdq) : nullptr;
    set_fp8_buffers(p, L, ws);
    return p;
}

FfnProblem shared_problem(const gbmoe_config* c, const void* x, const gbmoe_expert_weights* w, void* y, void* ws) {
    const Layout L = layout(c);
    FfnProblem p{};
    p.x = x; p.counts = nullptr; p.offsets = nullptr; p.sorted_pair = nullptr; p.pair_div = 1;
    p.E = 1; p.H = c->H; p.I = c->I_shared; p.n_rows = c->T;
    p.act_dtype = c->act_dtype; p.w_dtype = c->w_dtype;
    p.w_gate = w->w_gate; p.w_up = w->w_up; p.w_down = w->w_down;
    p.s_gate = w->s_gate; p.s_up = w->s_up; p.s_down = w->s_down;
    p.y = y;
    p.h = at<char>(ws, L.h); p.x_sorted = nullptr; p.sched = at<int32_t>(ws, L.sched);  // rows in order
    p.err = at<int32_t>(ws, L.err);
    p.w_dq = dequant_bytes(c, p.n_rows, p.E, p.I) ? at<char>(ws, L.wdq_sh) : nullptr;
    set_fp8_buffers(p, L, ws);
    return p;
}

// Every host-side check of moe_forward (x and out: the device buffers the
// layer reads and writes), so that a caller can run them before it enqueues
// anything of its own.
int check_forward(const gbmoe_config* cfg, const void* x, const void* w_router, const float* logit_bias,
                  const float* select_bias, const gbmoe_expert_weights* experts, const gbmoe_expert_weights* shared,
                  const void* out, const int32_t* topk_ids, const float* topk_w, const int32_t* counts_out, void* ws,
                  size_t ws_bytes) {
    int s = check_cfg(cfg);
    if (s) return s;
    if (cfg->T == 0) return check_ws(cfg, ws, ws_bytes);  // nothing to read or write
    if (!x || !w_router || !out || !aligned(x, 16) || !aligned(w_router, 16) || !aligned(out, 16))
        return GBMOE_EINVAL;
    if ((logit_bias && !aligned(logit_bias, 4)) || (select_bias && !aligned(select_bias, 4))) return GBMOE_EINVAL;
    if ((topk_ids && !aligned(topk_ids, 4)) || (topk_w && !aligned(topk_w, 4)) ||
        (counts_out && !aligned(counts_out, 4)))
        return GBMOE_EINVAL;
    if ((s = check_weights(cfg, experts))) return s;
    if (cfg->has_shared && (s = check_weights(cfg, shared))) return s;
    if ((s = check_ws(cfg, ws, ws_bytes))) return s;
    // every route must be launchable before anything is enqueued: the routed
    // problem with I, the shared one with I_shared
    if ((s = route_launchable(cfg, pick_route(cfg, (int64_t)cfg->T * cfg->top_k, cfg->E, cfg->I), cfg->I))) return s;
    if (cfg->has_shared && (s = route_launchable(cfg, pick_route(cfg, cfg->T, 1, cfg->I_shared), cfg->I_shared)))
        return s;
    return GBMOE_OK;
}

}  // namespace

extern "C" {

int gbmoe_last_cuda_error(void) {
    const int e = g_last_cuda_error;
    g_last_cuda_error = 0;
    return e;
}

const char* gbmoe_status_string(int s) {
    switch (s) {
        case GBMOE_OK: return "ok";
        case GBMOE_EINVAL: return "invalid argument";
        case GBMOE_EUNSUPPORTED: return "configuration not supported by the kernels";
        case GBMOE_EWORKSPACE: return "workspace too small";
        case GBMOE_ECUDA: return "CUDA launch or copy failed";
        case GBMOE_EDEVICE_TIMEOUT: return "device-side wait timed out";
        default: return "unknown status";
    }
}

int gbmoe_check_config(const gbmoe_config* cfg) { return check_cfg(cfg); }

size_t gbmoe_workspace_size(const gbmoe_config* cfg) {
    if (check_cfg(cfg) != GBMOE_OK) return 0;
    return layout(cfg).total;
}

int gbmoe_ffn_route(const gbmoe_config* cfg, int shared) {
    int s = check_cfg(cfg);
    if (s) return s;
    if (shared) return cfg->has_shared ? pick_route(cfg, cfg->T, 1, cfg->I_shared) : GBMOE_EINVAL;
    return pick_route(cfg, (int64_t)cfg->T * cfg->top_k, cfg->E, cfg->I);
}

int gbmoe_gate_route(const gbmoe_config* cfg) {
    int s = check_cfg(cfg);
    return s ? s : pick_gate(cfg);
}

int moe_rmsnorm(const gbmoe_config* cfg, const void* x, const void* gamma, float eps, void* y, void* stream) {
    int s = check_cfg(cfg);
    if (s) return s;
    if (!(eps >= 0.0f) || !std::isfinite(eps)) return GBMOE_EINVAL;
    if (cfg->T == 0) return GBMOE_OK;
    if (!x || !gamma || !y || !aligned(x, 16) || !aligned(gamma, 16) || !aligned(y, 16)) return GBMOE_EINVAL;
    const size_t bytes = (size_t)cfg->T * cfg->H * act_bytes(cfg->act_dtype);
    const char *xb = static_cast<const char*>(x), *yb = static_cast<const char*>(y);
    if (xb < yb + bytes && yb < xb + bytes) return GBMOE_EINVAL;  // overlapping rows
    return cuda_status(launch_rmsnorm(x, gamma, eps, cfg->T, cfg->H, cfg->act_dtype, y,
                                      static_cast<cudaStream_t>(stream)));
}

int moe_route(const gbmoe_config* cfg, const void* x, const void* w_router, const float* logit_bias,
              const float* select_bias, int32_t* topk_ids, float* topk_w, void* ws, size_t ws_bytes,
              void* stream) {
    int s = check_cfg(cfg);
    if (s) return s;
    if (cfg->T == 0) return check_ws(cfg, ws, ws_bytes);
    if (!x || !w_router || !topk_ids || !topk_w) return GBMOE_EINVAL;
    if (!aligned(x, 16) || !aligned(w_router, 16) || !aligned(topk_ids, 4) || !aligned(topk_w, 4))
        return GBMOE_EINVAL;
    if ((logit_bias && !aligned(logit_bias, 4)) || (select_bias && !aligned(select_bias, 4))) return GBMOE_EINVAL;
    if ((s = check_ws(cfg, ws, ws_bytes))) return s;
    const Layout L = layout(cfg);
    return cuda_status(launch_route(route_params(cfg), x, w_router, logit_bias, select_bias, at<float>(ws, L.logits),
                                    topk_ids, topk_w, route_scratch(cfg, ws), static_cast<cudaStream_t>(stream)));
}

int moe_permute(const gbmoe_config* cfg, const int32_t* topk_ids, int32_t* counts, int32_t* offsets,
                int32_t* sorted_pair, int32_t* pair_pos, void* ws, size_t ws_bytes, void* stream) {
    int s = check_cfg(cfg);
    if (s) return s;
    if (!topk_ids || !counts || !offsets || !sorted_pair || !pair_pos) return GBMOE_EINVAL;
    if (!aligned(topk_ids, 4) || !aligned(counts, 4) || !aligned(offsets, 4) || !aligned(sorted_pair, 4) ||
        !aligned(pair_pos, 4))
        return GBMOE_EINVAL;
    if ((s = check_ws(cfg, ws, ws_bytes))) return s;
    const Layout L = layout(cfg);
    return cuda_status(launch_permute(topk_ids, (int64_t)cfg->T * cfg->top_k, cfg->E, counts, offsets, sorted_pair,
                                      pair_pos, at<int32_t>(ws, L.perm), static_cast<cudaStream_t>(stream)));
}

int moe_grouped_ffn(const gbmoe_config* cfg, const void* x, const int32_t* counts, const int32_t* offsets,
                    const int32_t* sorted_pair, const gbmoe_expert_weights* experts, void* y_pairs, void* ws,
                    size_t ws_bytes, void* stream) {
    int s = check_cfg(cfg);
    if (s) return s;
    if (!x || !counts || !offsets || !sorted_pair || !y_pairs) return GBMOE_EINVAL;
    if (!aligned(x, 16) || !aligned(y_pairs, 16) || !aligned(counts, 4) || !aligned(offsets, 4) ||
        !aligned(sorted_pair, 4))
        return GBMOE_EINVAL;
    if ((s = check_weights(cfg, experts))) return s;
    if ((s = check_ws(cfg, ws, ws_bytes))) return s;
    if (cfg->T == 0) return GBMOE_OK;
    FfnProblem p = routed_problem(cfg, x, counts, offsets, sorted_pair, experts, y_pairs, ws);
    return run_ffn(cfg, p, pick_route(cfg, p.n_rows, cfg->E, cfg->I), static_cast<cudaStream_t>(stream));
}

int moe_shared_ffn(const gbmoe_config* cfg, const void* x, const gbmoe_expert_weights* shared, void* y_shared,
                   void* ws, size_t ws_bytes, void* stream) {
    int s = check_cfg(cfg);
    if (s) return s;
    if (!cfg->has_shared || !x || !y_shared || !aligned(x, 16) || !aligned(y_shared, 16)) return GBMOE_EINVAL;
    if ((s = check_weights(cfg, shared))) return s;
    if ((s = check_ws(cfg, ws, ws_bytes))) return s;
    if (cfg->T == 0) return GBMOE_OK;
    FfnProblem p = shared_problem(cfg, x, shared, y_shared, ws);
    return run_ffn(cfg, p, pick_route(cfg, cfg->T, 1, cfg->I_shared), static_cast<cudaStream_t>(stream));
}

int moe_combine(const gbmoe_config* cfg, const void* y_pairs, const float* topk_w, const int32_t* pair_pos,
                const void* y_shared, void* out, void* stream) {
    int s = check_cfg(cfg);
    if (s) return s;
    if (cfg->T == 0) return GBMOE_OK;
    if (!y_pairs || !topk_w || !pair_pos || !out) return GBMOE_EINVAL;
    if (!aligned(y_pairs, 16) || !aligned(out, 16) || !aligned(topk_w, 4) || !aligned(pair_pos, 4) ||
        (y_shared && !aligned(y_shared, 16)))
        return GBMOE_EINVAL;
    return cuda_status(launch_combine(y_pairs, topk_w, pair_pos, y_shared, out, cfg->T, cfg->top_k, cfg->H,
                                      cfg->act_dtype, static_cast<cudaStream_t>(stream)));
}

int moe_forward(const gbmoe_config* cfg, const void* x, const void* w_router, const float* logit_bias,
                const float* select_bias, const gbmoe_expert_weights* experts, const gbmoe_expert_weights* shared,
                void* out, int32_t* topk_ids, float* topk_w, int32_t* counts_out, void* ws, size_t ws_bytes,
                void* stream) {
    int s = check_forward(cfg, x, w_router, logit_bias, select_bias, experts, shared, out, topk_ids, topk_w,
                          counts_out, ws, ws_bytes);
    if (s || cfg->T == 0) return s;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const Layout L = layout(cfg);
    const int64_t P = (int64_t)cfg->T * cfg->top_k;
    const int r_routed = pick_route(cfg, P, cfg->E, cfg->I);
    const int r_shared = cfg->has_shared ? pick_route(cfg, cfg->T, 1, cfg->I_shared) : GBMOE_FFN_SIMT;
    if (const cudaError_t ce = cudaMemsetAsync(at<int32_t>(ws, L.err), 0, 4, st); ce != cudaSuccess) return cuda_status(ce);
    int32_t* ids = at<int32_t>(ws, L.ids);
    float* w = at<float>(ws, L.w);
    int32_t* counts = at<int32_t>(ws, L.counts);
    int32_t* offsets = at<int32_t>(ws, L.offsets);
    int32_t* sorted = at<int32_t>(ws, L.sorted);
    int32_t* pos = at<int32_t>(ws, L.pos);
    if ((s = cuda_status(launch_route(route_params(cfg), x, w_router, logit_bias, select_bias,
                                      at<float>(ws, L.logits), ids, w, route_scratch(cfg, ws), st))))
        return s;
    if ((s = cuda_status(launch_permute(ids, P, cfg->E, counts, offsets, sorted, pos, at<int32_t>(ws, L.perm), st))))
        return s;
    void* y = at<char>(ws, L.y);
    // the shared expert first: the routed down GEMM may fold the Weight Sum in
    void* ysh = nullptr;
    if (cfg->has_shared) {
        ysh = at<char>(ws, L.ysh);
        FfnProblem ps = shared_problem(cfg, x, shared, ysh, ws);
        if ((s = run_ffn(cfg, ps, r_shared, st))) return s;
    }
    FfnProblem pr = routed_problem(cfg, x, counts, offsets, sorted, experts, y, ws);
    const bool fused = cfg->combine_route == GBMOE_COMBINE_FUSED &&
                       bf16_gemm_route(r_routed);
    if (fused) {  // Weight Sum in the down GEMM's epilogue
        if ((s = cuda_status(cudaMemsetAsync(at<int32_t>(ws, L.arrive), 0, (size_t)cfg->T * (cfg->H / 256) * 4, st))))
            return s;
        pr.fuse_k = cfg->top_k;
        pr.topk_w = w;
        pr.y_shared = ysh;
        pr.out_final = out;
        pr.arrive = at<int32_t>(ws, L.arrive);
    }
    if ((s = run_ffn(cfg, pr, r_routed, st))) return s;
    if (!fused &&
        (s = cuda_status(launch_combine(y, w, pos, ysh, out, cfg->T, cfg->top_k, cfg->H, cfg->act_dtype, st))))
        return s;
    if (topk_ids && (s = cuda_status(cudaMemcpyAsync(topk_ids, ids, P * 4, cudaMemcpyDeviceToDevice, st)))) return s;
    if (topk_w && (s = cuda_status(cudaMemcpyAsync(topk_w, w, P * 4, cudaMemcpyDeviceToDevice, st)))) return s;
    if (counts_out &&
        (s = cuda_status(cudaMemcpyAsync(counts_out, counts, (size_t)cfg->E * 4, cudaMemcpyDeviceToDevice, st))))
        return s;
    return GBMOE_OK;
}

int moe_forward_hostio(const gbmoe_config* cfg, const void* x_host, const void* w_router, const float* logit_bias,
                       const float* select_bias, const gbmoe_expert_weights* experts,
                       const gbmoe_expert_weights* shared, void* out_host, void* ws, size_t ws_bytes, void* stream) {
    int s = check_cfg(cfg);
    if (s) return s;
    if ((s = check_ws(cfg, ws, ws_bytes))) return s;
    if (cfg->T == 0) return GBMOE_OK;
    if (!x_host || !out_host) return GBMOE_EINVAL;
    const Layout L = layout(cfg);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const size_t bytes = (size_t)cfg->T * cfg->H * act_bytes(cfg->act_dtype);
    void* xin = at<char>(ws, L.xin);
    void* xout = at<char>(ws, L.xout);
    // the layer's own checks first, so that a bad argument enqueues no copy
    if ((s = check_forward(cfg, xin, w_router, logit_bias, select_bias, experts, shared, xout, nullptr, nullptr,
                           nullptr, ws, ws_bytes)))
        return s;
    if (bytes && (s = cuda_status(cudaMemcpyAsync(xin, x_host, bytes, cudaMemcpyHostToDevice, st)))) return s;
    s = moe_forward(cfg, xin, w_router, logit_bias, select_bias, experts, shared, xout, nullptr, nullptr, nullptr, ws,
                    ws_bytes, stream);
    if (s) return s;
    if (bytes && (s = cuda_status(cudaMemcpyAsync(out_host, xout, bytes, cudaMemcpyDeviceToHost, st)))) return s;
    return GBMOE_OK;
}

int moe_device_status(void* ws, void* stream, int32_t* status) {
    if (!ws || !status || !aligned(ws, kAlign)) return GBMOE_EINVAL;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    int32_t word = 0;
    if (const cudaError_t ce = cudaStreamSynchronize(st); ce != cudaSuccess) return cuda_status(ce);
    if (const cudaError_t ce = cudaMemcpy(&word, ws, 4, cudaMemcpyDeviceToHost); ce != cudaSuccess) return cuda_status(ce);
    if (const cudaError_t ce = cudaMemset(ws, 0, 4); ce != cudaSuccess) return cuda_status(ce);
    *status = word ? GBMOE_EDEVICE_TIMEOUT : GBMOE_OK;
    return GBMOE_OK;
}

}  // extern "C"
