/*
 * CPU oracle for the MoE layer forward: MoE Gate -> Fused MoE -> Weight Sum.
 *
 * TEST INFRASTRUCTURE. Only the tests, the smoke check and the benchmark's
 * CPU-baseline leg use this file; the product library never links, loads or
 * calls it, and it shares no code, header or table with the CUDA path.
 *
 * What the paper fixes: the layer's semantic skeleton is the three nodes
 * MoE Gate, Fused MoE and Weight Sum (Fig. 1 in Section 1; Fig. 3 and its
 * discussion in Section 5.1), and the
 * model's mathematical semantics may not change under any implementation
 * route (Model Semantics Invariant, Section 3.3). It prints no formula for
 * any node. Each function below therefore writes out the standard definition
 * of its node in the plainest form, and states the reading it takes where the
 * paper is silent. Floating point is fp64 except where the result decides an
 * integer (the expert choice): there the decision is taken in fp32, in a fixed
 * operation order that the GPU path reproduces, so routing can be compared
 * bit for bit.
 *
 * Compile with -ffp-contract=off: every a*b+c below that is meant as one
 * rounding is written as fmaf(); everything else must round after each step.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* ----------------------------------------------------------- threading */

typedef void (*range_fn)(void* ctx, int64_t begin, int64_t end);
typedef struct { range_fn fn; void* ctx; int64_t begin, end; } job_t;

static int g_threads = 1;
void oracle_set_threads(int n) { g_threads = n < 1 ? 1 : (n > 256 ? 256 : n); }
int oracle_get_threads(void) { return g_threads; }

static void* job_main(void* p) {
    job_t* j = (job_t*)p;
    j->fn(j->ctx, j->begin, j->end);
    return NULL;
}

/* Splits [0, n) into contiguous ranges, one per thread. Work items are
 * independent, so the split never changes a result. */
static void parallel_for(int64_t n, range_fn fn, void* ctx) {
    int nt = g_threads;
    if (nt > n) nt = (int)(n > 0 ? n : 1);
    if (nt <= 1) { fn(ctx, 0, n); return; }
    pthread_t th[256];
    job_t jobs[256];
    int ok[256];
    int64_t chunk = (n + nt - 1) / nt;
    for (int t = 0; t < nt; ++t) {
        jobs[t].fn = fn; jobs[t].ctx = ctx;
        jobs[t].begin = t * chunk < n ? t * chunk : n;
        jobs[t].end = (t + 1) * chunk < n ? (t + 1) * chunk : n;
        ok[t] = pthread_create(&th[t], NULL, job_main, &jobs[t]) == 0;
        if (!ok[t]) fn(ctx, jobs[t].begin, jobs[t].end);
    }
    for (int t = 0; t < nt; ++t)
        if (ok[t]) pthread_join(th[t], NULL);
}

/* ============================================================ MoE Gate */

/*
 * Router logits l[t,e] = x[t,:] . Wg[e,:] (+ logit_bias[e]), in fp32.
 *
 * Reading (the paper gives no order): the dot product is split over 32
 * partial sums. Partial sum p (p = 0..31) takes the 8-element chunks
 * c = p, p+32, p+64, ... (chunk c covers elements 8c..8c+7) in increasing c
 * and, inside a chunk, increasing element, each step one fused multiply-add.
 * The 32 partial sums are then combined pairwise: at offset d = 16, 8, 4, 2, 1
 * every partial sum p becomes s[p] + s[p xor d]. Because one addition is
 * commutative, all 32 end equal, and that value is the logit. The bias is
 * then added with one fp32 addition. Requires H to be a multiple of 256.
 */
typedef struct {
    int64_t H, E;
    const float *x, *wg, *bias;
    float* logits;
} logit_ctx;

static float pinned_dot(const float* a, const float* b, int64_t H) {
    float s[32];
    for (int p = 0; p < 32; ++p) s[p] = 0.0f;
    for (int64_t c = 0; c < H / 8; ++c) {
        int p = (int)(c % 32);
        for (int i = 0; i < 8; ++i) s[p] = fmaf(a[8 * c + i], b[8 * c + i], s[p]);
    }
    for (int d = 16; d >= 1; d /= 2) {
        float n[32];
        for (int p = 0; p < 32; ++p) n[p] = s[p] + s[p ^ d];
        for (int p = 0; p < 32; ++p) s[p] = n[p];
    }
    return s[0];
}

static void logit_range(void* vp, int64_t b, int64_t e) {
    logit_ctx* c = (logit_ctx*)vp;
    for (int64_t t = b; t < e; ++t)
        for (int64_t x = 0; x < c->E; ++x) {
            float l = pinned_dot(c->x + t * c->H, c->wg + x * c->H, c->H);
            if (c->bias) l = l + c->bias[x];
            c->logits[t * c->E + x] = l;
        }
}

int oracle_gate_logits(int64_t T, int64_t H, int64_t E, const float* x, const float* wg,
                       const float* logit_bias, float* logits) {
    if (H % 256 != 0 || T < 0 || E < 1) return -1;
    logit_ctx c = {H, E, x, wg, logit_bias, logits};
    parallel_for(T, logit_range, &c);
    return 0;
}

/*
 * RMSNorm of the layer input before the gate (the step before the MoE Gate
 * node): y = x / sqrt(mean(x^2) + eps) * gamma, the standard definition.
 * Its result decides the expert choice (the logits are taken from it), so
 * it is computed in fp32 in a fixed order the GPU reproduces (reading: the
 * paper gives no formula): ss = sum of x^2 in the logits' order
 * (pinned_dot(x, x)); ms = ss / H; v = ms + eps; r = sqrt(v); inv = 1 / r;
 * y[h] = (x[h] * inv) * gamma[h]; every step one correctly rounded fp32
 * operation. The caller rounds y to the activation dtype.
 */
typedef struct {
    int64_t H;
    const float *x, *gamma;
    float eps;
    float* y;
} norm_ctx;

static void norm_range(void* vp, int64_t b, int64_t e) {
    norm_ctx* c = (norm_ctx*)vp;
    for (int64_t t = b; t < e; ++t) {
        const float* xr = c->x + t * c->H;
        const float ss = pinned_dot(xr, xr, c->H);
        const float ms = ss / (float)c->H;
        const float v = ms + c->eps;
        const float r = sqrtf(v);
        const float inv = 1.0f / r;
        for (int64_t h = 0; h < c->H; ++h) {
            const float xs = xr[h] * inv;
            c->y[t * c->H + h] = xs * c->gamma[h];
        }
    }
}

int oracle_rmsnorm(int64_t T, int64_t H, const float* x, const float* gamma, float eps, float* y) {
    if (H % 256 != 0 || T < 0 || !(eps >= 0.0f)) return -1;
    norm_ctx c = {H, x, gamma, eps, y};
    parallel_for(T, norm_range, &c);
    return 0;
}

/*
 * Pinned fp32 exponential, used where an exponential decides the expert
 * choice (sigmoid scores plus a selection bias). Written from the
 * mathematics, not from any library:
 *   a NaN is returned as it is; otherwise clamp x to [-86, 88] so that the
 *   result stays a normal number;
 *   n = rint(x * log2(e));  r = (x - n*ln2_hi) - n*ln2_lo  (Cody and Waite,
 *   "Software Manual for the Elementary Functions", 1980: ln2_hi keeps the
 *   leading 16 bits of ln 2 so that n*ln2_hi is exact);
 *   exp(r) by its Taylor series to degree 8, evaluated by Horner's rule with
 *   a separate multiply and add at each step (|r| <= 0.347, the truncation
 *   error is below 3e-10 relative);  result = p * 2^n built from exponent
 *   bits. Every step is one IEEE fp32 operation in this order.
 */
static float f32_from_bits(uint32_t u) { float f; memcpy(&f, &u, 4); return f; }

float oracle_pexp(float x) {
    const float log2e = f32_from_bits(0x3fb8aa3bu);  /* fp32(1/ln 2)           */
    const float ln2_hi = f32_from_bits(0x3f317200u); /* ln 2, 16 leading bits   */
    const float ln2_lo = f32_from_bits(0x35bfbe8eu); /* fp32(ln 2 - ln2_hi)     */
    static const uint32_t inv_fact[9] = {              /* fp32(1/i!), i = 0..8   */
        0x3f800000u, 0x3f800000u, 0x3f000000u, 0x3e2aaaabu, 0x3d2aaaabu,
        0x3c088889u, 0x3ab60b61u, 0x39500d01u, 0x37d00d01u};
    if (isnan(x)) return x; /* NaN in, NaN out, as for exp */
    if (x < -86.0f) x = -86.0f;
    if (x > 88.0f) x = 88.0f;
    float t = x * log2e;
    float n = rintf(t);
    float r = x - n * ln2_hi;
    r = r - n * ln2_lo;
    float p = f32_from_bits(inv_fact[8]);
    for (int i = 7; i >= 0; --i) {
        p = p * r;
        p = p + f32_from_bits(inv_fact[i]);
    }
    uint32_t bits = (uint32_t)((int32_t)n + 127) << 23;
    return p * f32_from_bits(bits);
}

/* Sigmoid score in fp32: s = 1 / (1 + pexp(-l)), IEEE division. */
float oracle_sigmoid(float l) {
    float d = 1.0f + oracle_pexp(-l);
    return 1.0f / d;
}

typedef struct {
    int32_t T, E, top_k;
    int32_t score;       /* 0 = softmax, 1 = sigmoid */
    int32_t renormalize; /* 1: weights over the selected experts sum to 1 (x scale) */
    int32_t n_group, topk_group;
    float routed_scale;
} oracle_route_cfg;

/* Key a score takes in the expert choice. Reading (the paper is silent on
 * non-finite scores): a NaN counts as -infinity, so that every comparison
 * below is a total order and the choice stays defined; ties, as always, go
 * to the lower index. */
static float choice_key(float v) { return isnan(v) ? -INFINITY : v; }

/* Index of the largest key among those with allowed[e] != 0; the lowest index
 * wins a tie (the scan is ascending and only a strictly larger key replaces). */
static int argmax_allowed(const float* key, const unsigned char* allowed, int n) {
    int best = -1;
    for (int e = 0; e < n; ++e) {
        if (!allowed[e]) continue;
        if (best < 0 || key[e] > key[best]) best = e;
    }
    return best;
}

/*
 * Expert selection and routing weights for every token.
 *
 * Softmax scoring (reading): the selection key is the logit itself (softmax
 * is increasing, so ordering by logit equals ordering by probability and no
 * exponential decides the choice). The top_k largest keys are taken in
 * descending order, equal keys going to the lower expert index. Weights, in
 * fp64: renormalised, w_j = exp(l_j - m) / sum over selected exp(l_i - m) with
 * m the largest selected logit; otherwise the full softmax over all E experts
 * evaluated at the selected ones. Both are multiplied by routed_scale.
 *
 * Sigmoid scoring with group-limited selection (reading, following the
 * DeepSeek-V3 description of this router): s_e = sigmoid(l_e) in fp32
 * (pinned exponential), q_e = s_e + select_bias[e] (fp32, bias used for the
 * choice only). Experts form n_group contiguous groups; a group's score is
 * the fp32 sum of its two largest q. The topk_group best groups are kept
 * (ties to the lower group), then the top_k largest q inside kept groups are
 * taken in descending order (ties to the lower expert). Weights, in fp64:
 * w_j = s_j / sum over selected s (renormalised) or s_j, times routed_scale.
 * With n_group = 1 the group step keeps every expert.
 *
 * ids[t*top_k + j] is the j-th selected expert, w[t*top_k + j] its weight.
 */
int oracle_route(const oracle_route_cfg* c, const float* logits, const float* select_bias,
                 int32_t* ids, double* w) {
    const int E = c->E, k = c->top_k;
    if (k < 1 || k > E) return -1;
    if (c->score == 1) {
        if (c->n_group < 1 || E % c->n_group) return -1;
        if (c->n_group > 1 && E / c->n_group < 2) return -1;
        if (c->topk_group < 1 || c->topk_group > c->n_group) return -1;
        if (k > c->topk_group * (E / c->n_group)) return -1;
    }
    float* key = (float*)malloc(sizeof(float) * E);
    float* s = (float*)malloc(sizeof(float) * E);
    unsigned char* allowed = (unsigned char*)malloc(E);
    const int G = c->n_group > 0 ? c->n_group : 1;
    float* gscore = (float*)malloc(sizeof(float) * G);
    unsigned char* gallowed = (unsigned char*)malloc(G);
    for (int64_t t = 0; t < c->T; ++t) {
        const float* l = logits + t * E;
        int32_t* id = ids + t * k;
        double* wt = w + t * k;
        if (c->score == 0) {
            for (int e = 0; e < E; ++e) { key[e] = choice_key(l[e]); allowed[e] = 1; }
        } else {
            for (int e = 0; e < E; ++e) {
                s[e] = oracle_sigmoid(l[e]);
                key[e] = choice_key(select_bias ? s[e] + select_bias[e] : s[e]);
                allowed[e] = 1;
            }
            if (G > 1) {
                const int gs = E / G;
                for (int g = 0; g < G; ++g) {
                    /* the two largest q of group g */
                    int a = -1, b = -1;
                    for (int e = g * gs; e < (g + 1) * gs; ++e) {
                        if (a < 0 || key[e] > key[a]) { b = a; a = e; }
                        else if (b < 0 || key[e] > key[b]) b = e;
                    }
                    gscore[g] = choice_key(key[a] + key[b]);
                    gallowed[g] = 1;
                }
                unsigned char* kept = (unsigned char*)calloc(G, 1);
                for (int r = 0; r < c->topk_group; ++r) {
                    int g = argmax_allowed(gscore, gallowed, G);
                    kept[g] = 1;
                    gallowed[g] = 0;
                }
                for (int e = 0; e < E; ++e) allowed[e] = kept[e / gs];
                free(kept);
            }
        }
        for (int j = 0; j < k; ++j) {
            int e = argmax_allowed(key, allowed, E);
            id[j] = e;
            allowed[e] = 0;
        }
        if (c->score == 0) {
            if (c->renormalize) {
                double m = (double)l[id[0]], z = 0.0;
                for (int j = 0; j < k; ++j) z += exp((double)l[id[j]] - m);
                for (int j = 0; j < k; ++j) wt[j] = exp((double)l[id[j]] - m) / z * c->routed_scale;
            } else {
                double m = (double)l[0], z = 0.0;
                for (int e = 1; e < E; ++e) if ((double)l[e] > m) m = (double)l[e];
                for (int e = 0; e < E; ++e) z += exp((double)l[e] - m);
                for (int j = 0; j < k; ++j) wt[j] = exp((double)l[id[j]] - m) / z * c->routed_scale;
            }
        } else {
            double z = 0.0;
            for (int j = 0; j < k; ++j) z += (double)s[id[j]];
            for (int j = 0; j < k; ++j)
                wt[j] = (c->renormalize ? (double)s[id[j]] / z : (double)s[id[j]]) * c->routed_scale;
        }
    }
    free(key); free(s); free(allowed); free(gscore); free(gallowed);
    return 0;
}

/* ============================================ Fused MoE: permutation */

/*
 * Groups the P = T*top_k (token, slot) pairs by expert. Pair p = t*top_k + j
 * goes to expert ids[p]. Reading (order unstated in the paper): a stable
 * counting sort, experts ascending and pairs ascending inside an expert.
 *   counts[e]      number of pairs routed to e
 *   offsets[e]     sum of counts[0..e-1] (offsets[E] = P)
 *   sorted_pair[r] the pair at sorted position r
 *   pair_pos[p]    the sorted position of pair p (inverse of sorted_pair)
 */
int oracle_permute(int64_t P, int32_t E, const int32_t* ids, int32_t* counts, int32_t* offsets,
                   int32_t* sorted_pair, int32_t* pair_pos) {
    for (int e = 0; e < E; ++e) counts[e] = 0;
    for (int64_t p = 0; p < P; ++p) {
        if (ids[p] < 0 || ids[p] >= E) return -1;
        counts[ids[p]] += 1;
    }
    offsets[0] = 0;
    for (int e = 0; e < E; ++e) offsets[e + 1] = offsets[e] + counts[e];
    int64_t r = 0;
    for (int e = 0; e < E; ++e)
        for (int64_t p = 0; p < P; ++p)
            if (ids[p] == e) {
                sorted_pair[r] = (int32_t)p;
                pair_pos[p] = (int32_t)r;
                ++r;
            }
    return 0;
}

/* ============================== Fused MoE: stored weight formats */

/*
 * FP8 E4M3 value of a byte (the OCP 8-bit floating point format, "fn"
 * variant): sign bit, 4 exponent bits with bias 7, 3 mantissa bits;
 * exponent field 0 gives subnormals m * 2^-9; no infinities; S.1111.111 is
 * NaN. Block-wise E4M3 expert weights are the format named in Section 6.2.
 */
double oracle_e4m3_value(uint8_t code) {
    int sign = code >> 7, ex = (code >> 3) & 0xf, m = code & 7;
    double v;
    if (ex == 15 && m == 7) return NAN;
    if (ex == 0) v = ldexp((double)m, -9);
    else v = ldexp(1.0 + m / 8.0, ex - 7);
    return sign ? -v : v;
}

/* Dequantised weight of one [N, K] expert matrix stored as e4m3 codes with
 * one fp32 scale per 128x128 block: W[n,k] = e4m3(q[n,k]) * s[n/128][k/128],
 * exact in fp64 (a 4-bit by 24-bit significand product). The 256 code values
 * are taken from oracle_e4m3_value once per call; rows are independent and
 * shared out over threads. */
typedef struct {
    int64_t K;
    const uint8_t* q;
    const float* s;
    double* out;
    double value[256];
} fp8_ctx;

static void fp8_rows(void* vp, int64_t b, int64_t e) {
    fp8_ctx* c = (fp8_ctx*)vp;
    const int64_t K = c->K;
    for (int64_t n = b; n < e; ++n)
        for (int64_t k = 0; k < K; ++k)
            c->out[n * K + k] = c->value[c->q[n * K + k]] * (double)c->s[(n / 128) * (K / 128) + k / 128];
}

void oracle_dequant_fp8_b128(int64_t N, int64_t K, const uint8_t* q, const float* s, double* out) {
    fp8_ctx c;
    c.K = K; c.q = q; c.s = s; c.out = out;
    for (int code = 0; code < 256; ++code) c.value[code] = oracle_e4m3_value((uint8_t)code);
    parallel_for(N, fp8_rows, &c);
}

static double bf16_value(uint16_t h) { return (double)f32_from_bits((uint32_t)h << 16); }

/* Dequantised weight of one [N, K] expert matrix stored as symmetric int4
 * (two's complement nibble, element 2i in the low nibble of byte i of a row)
 * with one bf16 scale per 128 consecutive k: W[n,k] = q[n,k] * s[n][k/128],
 * exact in fp64. Rows are shared out over threads. */
typedef struct {
    int64_t K;
    const uint8_t* q;
    const uint16_t* s;
    double* out;
} int4_ctx;

static void int4_rows(void* vp, int64_t b, int64_t e) {
    int4_ctx* c = (int4_ctx*)vp;
    const int64_t K = c->K;
    for (int64_t n = b; n < e; ++n)
        for (int64_t k = 0; k < K; ++k) {
            uint8_t byte = c->q[n * (K / 2) + k / 2];
            int v = (k % 2 == 0) ? (byte & 0xf) : (byte >> 4);
            if (v >= 8) v -= 16;
            c->out[n * K + k] = (double)v * bf16_value(c->s[n * (K / 128) + k / 128]);
        }
}

void oracle_dequant_int4_g128(int64_t N, int64_t K, const uint8_t* q, const uint16_t* s, double* out) {
    int4_ctx c = {K, q, s, out};
    parallel_for(N, int4_rows, &c);
}

/*
 * MXFP4 (OCP Microscaling Formats v1.0): the MXFP4 expert weights of the
 * DeepSeek reference path (Section 6.2). Each element is FP4 E2M1: sign bit 3,
 * a 2-bit exponent with bias 1 (bits 2-1) and one mantissa bit (bit 0);
 * exponent 0 is subnormal, m * 0.5; no infinities or NaN. Each block of 32
 * consecutive k shares an E8M0 scale: 2^(s - 127), s = 255 being NaN.
 */
double oracle_e2m1_value(uint8_t code) {
    int sign = (code >> 3) & 1, ex = (code >> 1) & 3, m = code & 1;
    double v = ex == 0 ? 0.5 * m : ldexp(1.0 + 0.5 * m, ex - 1);
    return sign ? -v : v;
}

double oracle_e8m0_value(uint8_t s) { return s == 255 ? NAN : ldexp(1.0, (int)s - 127); }

/* Dequantised weight of one [N, K] expert matrix stored as MXFP4: element
 * 2i in the low nibble of byte i of a row, scale s[n][k/32]:
 * W[n,k] = e2m1(q[n,k]) * 2^(s[n][k/32] - 127), exact in fp64. Rows are
 * shared out over threads. */
typedef struct {
    int64_t K;
    const uint8_t* q;
    const uint8_t* s;
    double* out;
    double value[16];
} mxfp4_ctx;

static void mxfp4_rows(void* vp, int64_t b, int64_t e) {
    mxfp4_ctx* c = (mxfp4_ctx*)vp;
    const int64_t K = c->K;
    for (int64_t n = b; n < e; ++n)
        for (int64_t k = 0; k < K; ++k) {
            uint8_t byte = c->q[n * (K / 2) + k / 2];
            int code = (k % 2 == 0) ? (byte & 0xf) : (byte >> 4);
            c->out[n * K + k] = c->value[code] * oracle_e8m0_value(c->s[n * (K / 32) + k / 32]);
        }
}

void oracle_dequant_mxfp4(int64_t N, int64_t K, const uint8_t* q, const uint8_t* s, double* out) {
    mxfp4_ctx c;
    c.K = K; c.q = q; c.s = s; c.out = out;
    for (int code = 0; code < 16; ++code) c.value[code] = oracle_e2m1_value((uint8_t)code);
    parallel_for(N, mxfp4_rows, &c);
}

void oracle_pexp_n(int64_t n, const float* in, float* out) {
    for (int64_t i = 0; i < n; ++i) out[i] = oracle_pexp(in[i]);
}

void oracle_sigmoid_n(int64_t n, const float* in, float* out) {
    for (int64_t i = 0; i < n; ++i) out[i] = oracle_sigmoid(in[i]);
}

typedef struct {
    const void* in;
    double* out;
} widen_ctx;

static void widen_f32_range(void* vp, int64_t b, int64_t e) {
    widen_ctx* c = (widen_ctx*)vp;
    for (int64_t i = b; i < e; ++i) c->out[i] = (double)((const float*)c->in)[i];
}

static void widen_bf16_range(void* vp, int64_t b, int64_t e) {
    widen_ctx* c = (widen_ctx*)vp;
    for (int64_t i = b; i < e; ++i) c->out[i] = bf16_value(((const uint16_t*)c->in)[i]);
}

void oracle_widen_f32(int64_t n, const float* in, double* out) {
    widen_ctx c = {in, out};
    parallel_for(n, widen_f32_range, &c);
}

void oracle_widen_bf16(int64_t n, const uint16_t* in, double* out) {
    widen_ctx c = {in, out};
    parallel_for(n, widen_bf16_range, &c);
}

/* ==================================================== Weight Sum */

/*
 * out[t,:] = sum over j of w[t,j] * y_pairs[pair_pos[t*k + j], :]
 *            (+ y_shared[t,:] when a shared expert is present, weight 1),
 * in fp64. y_pairs holds one expert output row per sorted pair position.
 */
typedef struct {
    int64_t k, H;
    const double *y_pairs, *w, *y_shared;
    const int32_t* pair_pos;
    double* out;
} combine_ctx;

static void combine_range(void* vp, int64_t b, int64_t e) {
    combine_ctx* c = (combine_ctx*)vp;
    const int64_t k = c->k, H = c->H;
    for (int64_t t = b; t < e; ++t)
        for (int64_t h = 0; h < H; ++h) {
            double acc = 0.0;
            for (int64_t j = 0; j < k; ++j)
                acc += c->w[t * k + j] * c->y_pairs[(int64_t)c->pair_pos[t * k + j] * H + h];
            if (c->y_shared) acc += c->y_shared[t * H + h];
            c->out[t * H + h] = acc;
        }
}

void oracle_combine(int64_t T, int64_t k, int64_t H, const double* y_pairs, const double* w,
                    const int32_t* pair_pos, const double* y_shared, double* out) {
    combine_ctx c = {k, H, y_pairs, w, y_shared, pair_pos, out};
    parallel_for(T, combine_range, &c);
}
