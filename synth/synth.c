/*
 * Seeded synthetic inputs for the MoE layer workloads.
 *
 * This module generates input tensors only (activations, router weights,
 * per-expert weights and their quantised storage forms). It holds none of the
 * layer's arithmetic: no routing, no dequantisation, no FFN. Both the CPU
 * oracle and the GPU path receive exactly the arrays produced here.
 *
 * Generator: a counter-based use of SplitMix64 (Steele, Lea & Flood,
 * "Fast splittable pseudorandom number generators", OOPSLA 2014). The
 * n-th output of a stream with key K is mix(K + n * GAMMA); element i of a
 * tensor draws outputs n = 2i+1 and 2i+2, so any element can be produced
 * independently of the others and in any order or thread split.
 *
 * Normal variates: Irwin-Hall sum of eight 16-bit uniforms taken from the two
 * 64-bit outputs, centred in integers (exact), converted to fp32 (exact, the
 * magnitude stays below 2^19) and multiplied once by sigma / std(sum), so
 * every machine gets identical bits. Storage dtype rounding is RNE.
 *
 * Quantised storage forms (the checkpoint formats the layer consumes):
 *   fp8 e4m3, 128x128 blocks: s = amax(block) / 448 (fp32), q = e4m3(w / s)
 *     with round-to-nearest-even and saturation to +-448; s = 1 if amax = 0.
 *   int4 symmetric, groups of 128 along K: s = bf16(amax(group) / 7),
 *     q = clamp(rne(w / s), -8, 7); two's complement nibbles, the even k in
 *     the low nibble; s = 1 if amax = 0.
 *   MXFP4 (OCP Microscaling Formats v1.0), blocks of 32 along K: shared
 *     scale X = 2^(floor(log2(amax)) - 2) stored as its E8M0 exponent
 *     (biased by 127; 2 is the largest exponent of FP4 E2M1), elements
 *     q = E2M1(w / X) rounded to nearest, ties to an even code, saturating
 *     at +-6; sign in bit 3, even k in the low nibble; X = 1 if amax = 0.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define GAMMA 0x9e3779b97f4a7c15ULL

static inline uint64_t mix64(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xbf58476d1ce4e5b9ULL;
    z = (z ^ (z >> 27)) * 0x94d049bb133111ebULL;
    return z ^ (z >> 31);
}

uint64_t synth_stream_key(uint64_t seed, uint64_t tensor_id) {
    return mix64(mix64(seed + GAMMA) ^ mix64((tensor_id + 1) * GAMMA));
}

/* Centred Irwin-Hall(8) integer for element i: range [-262140, 262140]. */
static inline int32_t ih8(uint64_t key, uint64_t i) {
    uint64_t a = mix64(key + (2 * i + 1) * GAMMA);
    uint64_t b = mix64(key + (2 * i + 2) * GAMMA);
    int32_t s = 0;
    for (int q = 0; q < 4; ++q) {
        s += (int32_t)((a >> (16 * q)) & 0xffffu);
        s += (int32_t)((b >> (16 * q)) & 0xffffu);
    }
    return s - 262140; /* 8 * 32767.5 */
}

/* fp32 multiplier that maps the centred sum to N(0, sigma^2). */
static float sigma_scale(double sigma) {
    /* var of one 16-bit uniform = (65536^2 - 1) / 12; eight of them. */
    double sd = sqrt(8.0 * (65536.0 * 65536.0 - 1.0) / 12.0);
    return (float)(sigma / sd);
}

static inline float normal_f32(uint64_t key, uint64_t i, float scale) {
    return (float)ih8(key, i) * scale;
}

static inline uint16_t f32_to_bf16_rne(float f) {
    uint32_t u;
    memcpy(&u, &f, 4);
    if ((u & 0x7fffffffu) > 0x7f800000u) return (uint16_t)((u >> 16) | 0x40u);
    u += 0x7fffu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
}

static inline float bf16_to_f32(uint16_t h) {
    uint32_t u = (uint32_t)h << 16;
    float f;
    memcpy(&f, &u, 4);
    return f;
}

/* fp32 -> e4m3 (bias 7, no inf, max 448), round to nearest even, saturating. */
static uint8_t f32_to_e4m3(float f) {
    uint32_t u;
    memcpy(&u, &f, 4);
    uint8_t sign = (uint8_t)((u >> 24) & 0x80u);
    double a = fabs((double)f);
    if (a != a) return (uint8_t)(sign | 0x7f);
    if (a >= 448.0) return (uint8_t)(sign | 0x7e);
    if (a < 0.015625) { /* below 2^-6: subnormal step 2^-9 */
        int m = (int)nearbyint(a * 512.0); /* 8 lands on the smallest normal */
        return (uint8_t)(sign | m);
    }
    int ex;
    frexp(a, &ex);
    int e = ex - 1; /* a in [2^e, 2^(e+1)) */
    int m = (int)nearbyint((ldexp(a, -e) - 1.0) * 8.0);
    if (m == 8) { m = 0; e += 1; }
    return (uint8_t)(sign | ((e + 7) << 3) | m);
}

/* ---------------------------------------------------------------- threads */

typedef void (*range_fn)(void* ctx, int64_t begin, int64_t end);
typedef struct { range_fn fn; void* ctx; int64_t begin, end; } job_t;

static void* job_main(void* p) {
    job_t* j = (job_t*)p;
    j->fn(j->ctx, j->begin, j->end);
    return NULL;
}

static int g_threads = 0;
void synth_set_threads(int n) { g_threads = n; }

static void parallel_for(int64_t n, range_fn fn, void* ctx) {
    int nt = g_threads > 0 ? g_threads : 1;
    if (nt > 256) nt = 256;
    if (n < 4096 || nt == 1) { fn(ctx, 0, n); return; }
    if (nt > n) nt = (int)n;
    pthread_t th[256];
    job_t jobs[256];
    int64_t chunk = (n + nt - 1) / nt;
    for (int t = 0; t < nt; ++t) {
        jobs[t].fn = fn; jobs[t].ctx = ctx;
        jobs[t].begin = t * chunk;
        jobs[t].end = (t + 1) * chunk < n ? (t + 1) * chunk : n;
        if (jobs[t].begin >= jobs[t].end) continue;
        if (pthread_create(&th[t], NULL, job_main, &jobs[t]) != 0) {
            fn(ctx, jobs[t].begin, jobs[t].end);
            jobs[t].begin = jobs[t].end = 0;
        }
    }
    for (int t = 0; t < nt; ++t)
        if (jobs[t].begin < jobs[t].end) pthread_join(th[t], NULL);
}

/* ------------------------------------------------------- dense tensors */

typedef struct { uint64_t key; float scale; uint64_t offset; void* out; } dense_ctx;

static void dense_f32_range(void* p, int64_t b, int64_t e) {
    dense_ctx* c = (dense_ctx*)p;
    float* o = (float*)c->out;
    for (int64_t i = b; i < e; ++i) o[i] = normal_f32(c->key, c->offset + (uint64_t)i, c->scale);
}

static void dense_bf16_range(void* p, int64_t b, int64_t e) {
    dense_ctx* c = (dense_ctx*)p;
    uint16_t* o = (uint16_t*)c->out;
    for (int64_t i = b; i < e; ++i)
        o[i] = f32_to_bf16_rne(normal_f32(c->key, c->offset + (uint64_t)i, c->scale));
}

/* Elements [offset, offset + n) of the N(0, sigma^2) stream (seed, tensor_id). */
void synth_normal_f32(uint64_t seed, uint64_t tensor_id, double sigma, uint64_t offset,
                      int64_t n, float* out) {
    dense_ctx c = {synth_stream_key(seed, tensor_id), sigma_scale(sigma), offset, out};
    parallel_for(n, dense_f32_range, &c);
}

/* Same stream rounded to bf16 (RNE), stored as raw 16-bit patterns. */
void synth_normal_bf16(uint64_t seed, uint64_t tensor_id, double sigma, uint64_t offset,
                       int64_t n, uint16_t* out) {
    dense_ctx c = {synth_stream_key(seed, tensor_id), sigma_scale(sigma), offset, out};
    parallel_for(n, dense_bf16_range, &c);
}

/* ------------------------------------------------ fp8 e4m3, 128x128 blocks */

typedef struct {
    uint64_t key; float scale; int64_t N, K; int64_t e0;
    uint8_t* q; float* s;
} fp8_ctx;

static void fp8_range(void* p, int64_t b, int64_t e) {
    fp8_ctx* c = (fp8_ctx*)p;
    const int64_t nb = c->N / 128, kb = c->K / 128;
    float* tile = (float*)malloc(sizeof(float) * 128 * 128);
    for (int64_t blk = b; blk < e; ++blk) {
        int64_t ex = blk / (nb * kb), r = blk % (nb * kb);
        int64_t bn = r / kb, bk = r % kb;
        float amax = 0.0f;
        for (int i = 0; i < 128; ++i)
            for (int j = 0; j < 128; ++j) {
                int64_t n = bn * 128 + i, k = bk * 128 + j;
                uint64_t idx = (uint64_t)(((c->e0 + ex) * c->N + n) * c->K + k);
                float v = normal_f32(c->key, idx, c->scale);
                tile[i * 128 + j] = v;
                float av = fabsf(v);
                if (av > amax) amax = av;
            }
        float s = amax > 0.0f ? amax / 448.0f : 1.0f;
        c->s[blk] = s;
        for (int i = 0; i < 128; ++i)
            for (int j = 0; j < 128; ++j) {
                int64_t n = bn * 128 + i, k = bk * 128 + j;
                c->q[(ex * c->N + n) * c->K + k] = f32_to_e4m3(tile[i * 128 + j] / s);
            }
    }
    free(tile);
}

/* Experts [e0, e0+ne) of a [E, N, K] weight drawn from N(0, sigma^2) and stored
 * as e4m3 codes q [ne, N, K] with fp32 block scales s [ne, N/128, K/128].
 * Returns -1 unless N and K are multiples of 128. */
int synth_fp8_b128(uint64_t seed, uint64_t tensor_id, double sigma, int64_t e0, int64_t ne,
                   int64_t N, int64_t K, uint8_t* q, float* s) {
    if (N % 128 || K % 128) return -1;
    fp8_ctx c = {synth_stream_key(seed, tensor_id), sigma_scale(sigma), N, K, e0, q, s};
    parallel_for(ne * (N / 128) * (K / 128), fp8_range, &c);
    return 0;
}

/* --------------------------------------------- int4, groups of 128 along K */

typedef struct {
    uint64_t key; float scale; int64_t N, K; int64_t e0;
    uint8_t* q; uint16_t* s;
} int4_ctx;

static void int4_range(void* p, int64_t b, int64_t e) {
    int4_ctx* c = (int4_ctx*)p;
    const int64_t kg = c->K / 128;
    float g[128];
    for (int64_t grp = b; grp < e; ++grp) {
        int64_t row = grp / kg, gk = grp % kg; /* row = ex * N + n */
        int64_t ex = row / c->N, n = row % c->N;
        float amax = 0.0f;
        for (int j = 0; j < 128; ++j) {
            uint64_t idx = (uint64_t)(((c->e0 + ex) * c->N + n) * c->K + gk * 128 + j);
            g[j] = normal_f32(c->key, idx, c->scale);
            float av = fabsf(g[j]);
            if (av > amax) amax = av;
        }
        uint16_t sb = amax > 0.0f ? f32_to_bf16_rne(amax / 7.0f) : (uint16_t)0x3f80u;
        float sf = bf16_to_f32(sb);
        c->s[grp] = sb;
        uint8_t* dst = c->q + row * (c->K / 2) + gk * 64;
        for (int j = 0; j < 128; j += 2) {
            int q0 = (int)nearbyintf(g[j] / sf), q1 = (int)nearbyintf(g[j + 1] / sf);
            q0 = q0 < -8 ? -8 : (q0 > 7 ? 7 : q0);
            q1 = q1 < -8 ? -8 : (q1 > 7 ? 7 : q1);
            dst[j / 2] = (uint8_t)((q0 & 0xf) | ((q1 & 0xf) << 4));
        }
    }
}

/* Experts [e0, e0+ne) of a [E, N, K] weight drawn from N(0, sigma^2) and stored
 * as packed int4 q [ne, N, K/2] with bf16 group scales s [ne, N, K/128].
 * Returns -1 unless K is a multiple of 128. */
int synth_int4_g128(uint64_t seed, uint64_t tensor_id, double sigma, int64_t e0, int64_t ne,
                    int64_t N, int64_t K, uint8_t* q, uint16_t* s) {
    if (K % 128) return -1;
    int4_ctx c = {synth_stream_key(seed, tensor_id), sigma_scale(sigma), N, K, e0, q, s};
    parallel_for(ne * N * (K / 128), int4_range, &c);
    return 0;
}

/* ------------------------------------- MXFP4: E2M1 + E8M0 per 32 along K */

/* Magnitude code (0..7) of FP4 E2M1 nearest to a >= 0, ties to the even
 * code, saturating at 6. Grid: 0, 0.5, 1, 1.5, 2, 3, 4, 6. */
static int e2m1_code(double a) {
    static const double grid[8] = {0.0, 0.5, 1.0, 1.5, 2.0, 3.0, 4.0, 6.0};
    if (a >= 6.0) return 7;
    int best = 0;
    for (int c = 1; c < 8; ++c) {
        double d = fabs(a - grid[c]), db = fabs(a - grid[best]);
        if (d < db || (d == db && (c & 1) == 0)) best = c;
    }
    return best;
}

typedef struct {
    uint64_t key; float scale; int64_t N, K; int64_t e0;
    uint8_t* q; uint8_t* s;
} mxfp4_ctx;

static void mxfp4_range(void* p, int64_t b, int64_t e) {
    mxfp4_ctx* c = (mxfp4_ctx*)p;
    const int64_t kg = c->K / 32;
    float g[32];
    for (int64_t blk = b; blk < e; ++blk) {
        int64_t row = blk / kg, gk = blk % kg; /* row = ex * N + n */
        int64_t ex = row / c->N, n = row % c->N;
        float amax = 0.0f;
        for (int j = 0; j < 32; ++j) {
            uint64_t idx = (uint64_t)(((c->e0 + ex) * c->N + n) * c->K + gk * 32 + j);
            g[j] = normal_f32(c->key, idx, c->scale);
            float av = fabsf(g[j]);
            if (av > amax) amax = av;
        }
        int ex2 = 0; /* scale exponent: floor(log2(amax)) - 2 */
        if (amax > 0.0f) {
            int fe;
            frexp((double)amax, &fe); /* amax in [2^(fe-1), 2^fe) */
            ex2 = (fe - 1) - 2;
        }
        int biased = ex2 + 127;
        if (biased < 0) biased = 0;
        if (biased > 254) biased = 254;
        c->s[blk] = (uint8_t)biased;
        const double X = ldexp(1.0, biased - 127);
        uint8_t* dst = c->q + row * (c->K / 2) + gk * 16;
        for (int j = 0; j < 32; j += 2) {
            int n0 = e2m1_code(fabs((double)g[j]) / X) | (g[j] < 0.0f ? 8 : 0);
            int n1 = e2m1_code(fabs((double)g[j + 1]) / X) | (g[j + 1] < 0.0f ? 8 : 0);
            dst[j / 2] = (uint8_t)(n0 | (n1 << 4));
        }
    }
}

/* Experts [e0, e0+ne) of a [E, N, K] weight drawn from N(0, sigma^2) and stored
 * as MXFP4: packed E2M1 q [ne, N, K/2] (even k in the low nibble) with E8M0
 * block scales s [ne, N, K/32]. Returns -1 unless K is a multiple of 32. */
int synth_mxfp4(uint64_t seed, uint64_t tensor_id, double sigma, int64_t e0, int64_t ne, int64_t N,
                int64_t K, uint8_t* q, uint8_t* s) {
    if (K % 32) return -1;
    mxfp4_ctx c = {synth_stream_key(seed, tensor_id), sigma_scale(sigma), N, K, e0, q, s};
    parallel_for(ne * N * (K / 32), mxfp4_range, &c);
    return 0;
}
