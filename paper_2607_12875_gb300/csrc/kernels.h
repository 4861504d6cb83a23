// Internal launch interface between the C ABI (api.cu) and the kernels.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace gbmoe {

struct RouteParams {
    int T, H, E, top_k;
    int score, renormalize, n_group, topk_group;
    float routed_scale;
    int act_dtype;
    int gate_tc;  // 1: logits on the tensor cores, audited against the fixed order
};

// scratch of the tensor-core gate: schedule ints for T rows, the device error
// word, two words for the audit (max router row norm, count of flagged
// tokens) and the list of flagged tokens [T]
struct RouteScratch {
    int32_t* sched;
    int32_t* err;
    float* audit;
    int32_t* flagged;
};

// logits [T, E] fp32 scratch; topk_ids, topk_w [T, k]
cudaError_t launch_route(const RouteParams& rp, const void* x, const void* w_router, const float* logit_bias,
                         const float* select_bias, float* logits, int32_t* topk_ids, float* topk_w,
                         const RouteScratch& rs, cudaStream_t stream);
// RMSNorm of x [T, H] (act dtype) with gamma [H] into y, in the gate's order
cudaError_t launch_rmsnorm(const void* x, const void* gamma, float eps, int T, int H, int act_dtype, void* y,
                           cudaStream_t stream);
// router logits on the tensor cores (bf16 x and router weight; ffn_tc.cu)
cudaError_t launch_gate_tc(const void* x, const void* wg, const float* bias, float* logits, int T, int H, int E,
                           int32_t* sched, int32_t* err, cudaStream_t stream);

// Number of 1024-pair blocks the permutation uses, and its scratch ints.
int permute_blocks(int64_t P);
size_t permute_scratch_ints(int64_t P, int E);
cudaError_t launch_permute(const int32_t* topk_ids, int64_t P, int E, int32_t* counts, int32_t* offsets,
                           int32_t* sorted_pair, int32_t* pair_pos, int32_t* scratch, cudaStream_t stream);

// One grouped FFN problem: rows r of expert e are offsets[e] .. offsets[e+1]-1,
// the token of row r is sorted_pair[r] / pair_div (r itself when sorted_pair
// is null). counts null means one expert with n_rows rows.
struct FfnProblem {
    const void* x;              // [T, H] act
    const int32_t* counts;      // [E] or null
    const int32_t* offsets;     // [E+1] or null (then 0, n_rows)
    const int32_t* sorted_pair; // [rows] or null
    int pair_div;
    int E, H, I;
    int64_t n_rows;             // upper bound on rows (P, or T for the shared expert)
    int act_dtype, w_dtype;
    const void *w_gate, *w_up, *w_down, *s_gate, *s_up, *s_down;
    void* y;                    // [n_rows, H] act
    // scratch carved by the caller
    void* h;                    // [n_rows, I] act
    void* x_sorted;             // [n_rows, H] act: the sorted copy the quantised-weight one-CTA GEMM and the
                                // CTA-pair GEMMs read (null on routes that do not use one)
    void* w_dq;                 // bf16 [E, I, H] gate, [E, I, H] up, [E, H, I] down, or null:
                                // quantised weights are then decoded once into it (TC_DEQUANT)
    void* a_q;                  // fp8 route (TC_FP8): x rows in sorted order as two e4m3 code planes
                                //   [2, n_rows, H] (value and residual)
    float* a_s;                 //   and their 1x128 scales [n_rows, H/128]
    void* h_q;                  //   h the same way, [2, n_rows, I]
    float* h_s;                 //   and its 1x128 scales [n_rows, I/128]
    int cta_pair;               // tensor-core routes: 1 = CTA pairs (cta_group::2, 256-row M tiles)
    int32_t* sched;             // schedule ints, ffn_sched_ints(E, n_rows)
    int32_t* err;               // device error word
    // Weight Sum fused into the down GEMM (tensor-core routes; fuse_k = top_k,
    // 0 = off): y then receives topk_w[p] * y of pair p at row p (pair order)
    // and out_final[t] = sum_j slots of t (+ y_shared[t]); arrive holds
    // T * (H / 256) zeroed counters
    int fuse_k;
    const float* topk_w;
    const void* y_shared;
    void* out_final;
    int32_t* arrive;
};

size_t ffn_sched_ints(int E, int64_t n_rows);
constexpr int64_t kDequantRowsPerExpert = 256;  // AUTO: TC_DEQUANT from this many rows per expert
constexpr int64_t kPairRowsPerExpert = 1024;    // AUTO: CTA pairs from this many rows per expert
cudaError_t launch_ffn_stream(const FfnProblem& p, cudaStream_t stream);
size_t stream_smem_bytes(int act_dtype, int H, int I);  // per CTA, streaming route
// dynamic shared memory a CTA may use on sm_103a (227 KB); a streaming problem
// runs when its stream_smem_bytes fits
constexpr size_t stream_smem_budget() { return 227 * 1024; }
cudaError_t launch_ffn_simt(const FfnProblem& p, cudaStream_t stream);
cudaError_t launch_ffn_tc(const FfnProblem& p, cudaStream_t stream);
bool ffn_tc_supported(const FfnProblem& p);
bool ffn_tc_pair_supported(const FfnProblem& p);
cudaError_t launch_ffn_tc_fp8(const FfnProblem& p, cudaStream_t stream);
bool ffn_tc_fp8_supported(const FfnProblem& p);

cudaError_t launch_combine(const void* y_pairs, const float* topk_w, const int32_t* pair_pos, const void* y_shared,
                           void* out, int T, int k, int H, int act_dtype, cudaStream_t stream);

}  // namespace gbmoe
