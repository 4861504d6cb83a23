// Stored expert-weight formats: element access and 16-byte chunk decoding.
//   F32 / BF16       plain values
//   FP8_E4M3_B128    e4m3 bytes, fp32 scale per 128x128 block of the [N, K] matrix
//   INT4_G128        two's complement nibbles (even k low), bf16 scale per 128 k of a row
//   MXFP4            E2M1 nibbles (even k low), E8M0 scale per 32 k of a row
#pragma once

#include "common.cuh"

namespace gbmoe {

template <int WQ>
struct WFmt;

template <>
struct WFmt<GBMOE_F32> {
    static constexpr int CE = 8;   // elements per chunk
    static constexpr int NV = 2;   // 16-byte vectors per chunk
    __device__ static size_t row_bytes(int K) { return (size_t)K * 4; }
    __device__ static const void* scale_row(const void*, int64_t, int, int, int) { return nullptr; }
    __device__ static float scale_at(const void*, int) { return 1.0f; }
    __device__ __forceinline__ static void decode8(const uint4 (&r)[NV], int sub, float, float (&w)[8]) {
        (void)sub;
        w[0] = __uint_as_float(r[0].x); w[1] = __uint_as_float(r[0].y);
        w[2] = __uint_as_float(r[0].z); w[3] = __uint_as_float(r[0].w);
        w[4] = __uint_as_float(r[1].x); w[5] = __uint_as_float(r[1].y);
        w[6] = __uint_as_float(r[1].z); w[7] = __uint_as_float(r[1].w);
    }
    __device__ static float elem(const void* w, const void*, int64_t e, int N, int K, int n, int k) {
        return static_cast<const float*>(w)[((size_t)e * N + n) * K + k];
    }
};

template <>
struct WFmt<GBMOE_BF16> {
    static constexpr int CE = 8;
    static constexpr int NV = 1;
    __device__ static size_t row_bytes(int K) { return (size_t)K * 2; }
    __device__ static const void* scale_row(const void*, int64_t, int, int, int) { return nullptr; }
    __device__ static float scale_at(const void*, int) { return 1.0f; }
    __device__ __forceinline__ static void decode8(const uint4 (&r)[NV], int, float, float (&w)[8]) {
        w[0] = bf16lo(r[0].x); w[1] = bf16hi(r[0].x); w[2] = bf16lo(r[0].y); w[3] = bf16hi(r[0].y);
        w[4] = bf16lo(r[0].z); w[5] = bf16hi(r[0].z); w[6] = bf16lo(r[0].w); w[7] = bf16hi(r[0].w);
    }
    __device__ static float elem(const void* w, const void*, int64_t e, int N, int K, int n, int k) {
        return __bfloat162float(static_cast<const __nv_bfloat16*>(w)[((size_t)e * N + n) * K + k]);
    }
};

template <>
struct WFmt<GBMOE_FP8_E4M3_B128> {
    static constexpr int CE = 16;
    static constexpr int NV = 1;
    __device__ static size_t row_bytes(int K) { return (size_t)K; }
    // scale of element (n, k) of expert e's [N, K] matrix
    __device__ static float scale(const void* s, int64_t e, int N, int K, int n, int k) {
        return static_cast<const float*>(s)[((size_t)e * (N / 128) + n / 128) * (K / 128) + k / 128];
    }
    // scales along k of row n, and the one covering element k
    __device__ static const void* scale_row(const void* s, int64_t e, int N, int K, int n) {
        return static_cast<const float*>(s) + ((size_t)e * (N / 128) + n / 128) * (K / 128);
    }
    __device__ static float scale_at(const void* row, int k) { return static_cast<const float*>(row)[k / 128]; }
    __device__ __forceinline__ static void decode8(const uint4 (&r)[NV], int sub, float sc, float (&w)[8]) {
        const uint32_t lo = sub ? r[0].z : r[0].x, hi = sub ? r[0].w : r[0].y;
        const float2 a = e4m3x2_to_f32x2(lo & 0xffffu), b = e4m3x2_to_f32x2(lo >> 16);
        const float2 c = e4m3x2_to_f32x2(hi & 0xffffu), d = e4m3x2_to_f32x2(hi >> 16);
        w[0] = a.x * sc; w[1] = a.y * sc; w[2] = b.x * sc; w[3] = b.y * sc;
        w[4] = c.x * sc; w[5] = c.y * sc; w[6] = d.x * sc; w[7] = d.y * sc;
    }
    __device__ static float elem(const void* w, const void* s, int64_t e, int N, int K, int n, int k) {
        uint32_t b = static_cast<const uint8_t*>(w)[((size_t)e * N + n) * K + k];
        return e4m3_to_f32(b) * scale(s, e, N, K, n, k);
    }
};

template <>
struct WFmt<GBMOE_INT4_G128> {
    static constexpr int CE = 32;
    static constexpr int NV = 1;
    __device__ static size_t row_bytes(int K) { return (size_t)K / 2; }
    __device__ static float scale(const void* s, int64_t e, int N, int K, int n, int k) {
        return __bfloat162float(static_cast<const __nv_bfloat16*>(s)[((size_t)e * N + n) * (K / 128) + k / 128]);
    }
    __device__ static const void* scale_row(const void* s, int64_t e, int N, int K, int n) {
        return static_cast<const __nv_bfloat16*>(s) + ((size_t)e * N + n) * (K / 128);
    }
    __device__ static float scale_at(const void* row, int k) {
        return __bfloat162float(static_cast<const __nv_bfloat16*>(row)[k / 128]);
    }
    __device__ __forceinline__ static void decode8(const uint4 (&r)[NV], int sub, float sc, float (&w)[8]) {
        uint32_t v = sub == 0 ? r[0].x : sub == 1 ? r[0].y : sub == 2 ? r[0].z : r[0].w;
#pragma unroll
        for (int i = 0; i < 8; ++i) w[i] = int4_to_f32((v >> (4 * i)) & 0xfu) * sc;
    }
    __device__ static float elem(const void* w, const void* s, int64_t e, int N, int K, int n, int k) {
        uint32_t b = static_cast<const uint8_t*>(w)[((size_t)e * N + n) * (K / 2) + k / 2];
        uint32_t nib = (k & 1) ? (b >> 4) : (b & 0xfu);
        return int4_to_f32(nib) * scale(s, e, N, K, n, k);
    }
};

template <>
struct WFmt<GBMOE_MXFP4> {
    static constexpr int CE = 32;  // one 16-byte chunk = one 32-element scale block
    static constexpr int NV = 1;
    __device__ static size_t row_bytes(int K) { return (size_t)K / 2; }
    __device__ static float scale(const void* s, int64_t e, int N, int K, int n, int k) {
        return e8m0_to_f32(static_cast<const uint8_t*>(s)[((size_t)e * N + n) * (K / 32) + k / 32]);
    }
    __device__ static const void* scale_row(const void* s, int64_t e, int N, int K, int n) {
        return static_cast<const uint8_t*>(s) + ((size_t)e * N + n) * (K / 32);
    }
    __device__ static float scale_at(const void* row, int k) {
        return e8m0_to_f32(static_cast<const uint8_t*>(row)[k / 32]);
    }
    __device__ __forceinline__ static void decode8(const uint4 (&r)[NV], int sub, float sc, float (&w)[8]) {
        uint32_t v = sub == 0 ? r[0].x : sub == 1 ? r[0].y : sub == 2 ? r[0].z : r[0].w;
#pragma unroll
        for (int i = 0; i < 8; ++i) w[i] = e2m1_to_f32((v >> (4 * i)) & 0xfu) * sc;
    }
    __device__ static float elem(const void* w, const void* s, int64_t e, int N, int K, int n, int k) {
        uint32_t b = static_cast<const uint8_t*>(w)[((size_t)e * N + n) * (K / 2) + k / 2];
        uint32_t nib = (k & 1) ? (b >> 4) : (b & 0xfu);
        return e2m1_to_f32(nib) * scale(s, e, N, K, n, k);
    }
};

}  // namespace gbmoe
