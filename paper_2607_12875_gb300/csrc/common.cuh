// Shared device helpers for the MoE layer kernels (sm_103a).
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>

#include "../../include/gbmoe.h"

namespace gbmoe {

constexpr int kWarp = 32;

__host__ __device__ __forceinline__ int64_t min64(int64_t a, int64_t b) { return a < b ? a : b; }

// ------------------------------------------- programmatic dependent launch
//
// Every kernel of the layer starts with pdl_enter(): it waits until the
// kernel before it on the stream has completed and its writes are visible,
// and only then lets the next kernel be scheduled. So at most two adjacent
// kernels are resident at once, the later one parked at its wait: the next
// launch's scheduling overlaps this kernel's run, and no data hazard opens.
// Without a programmatic predecessor both instructions return at once.
__device__ __forceinline__ void pdl_enter() {
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Launch with programmatic stream serialization allowed (see pdl_enter).
template <typename... KArgs, typename... Args>
cudaError_t launch_k(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                     Args&&... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args&&>(args)...);
}

// The same with clusters of `cluster_x` CTAs along x (grid.x a multiple of it).
template <typename... KArgs, typename... Args>
cudaError_t launch_k_cluster(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                             int cluster_x, Args&&... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = (unsigned)cluster_x;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args&&>(args)...);
}

// Clusters of `cluster_x` CTAs of this kernel (block threads, smem bytes)
// that can be resident at once on the current device, or 0 on error.
template <typename... KArgs>
int max_active_clusters(void (*kernel)(KArgs...), int threads, size_t smem, int cluster_x) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)cluster_x);
    cfg.blockDim = dim3((unsigned)threads);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = (unsigned)cluster_x;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, reinterpret_cast<const void*>(kernel), &cfg) != cudaSuccess) {
        (void)cudaGetLastError();
        return 0;
    }
    return n;
}

// ------------------------------------------------- per-device host state

constexpr int kMaxDevices = 64;

// Runs a setup step (a cudaFuncSetAttribute, say) once per device: run(f)
// calls f only while it has not yet succeeded on the current device. Two
// threads racing on the first call may both run f, which is harmless for the
// idempotent steps it is used for.
struct DeviceOnce {
    std::atomic<uint64_t> done{0};
    template <typename F>
    cudaError_t run(F&& f) {
        int dev = 0;
        if (cudaError_t e = cudaGetDevice(&dev); e != cudaSuccess) return e;
        const uint64_t bit = dev >= 0 && dev < kMaxDevices ? 1ull << dev : 0;
        if (bit && (done.load(std::memory_order_acquire) & bit)) return cudaSuccess;
        const cudaError_t e = f();
        if (e == cudaSuccess && bit) done.fetch_or(bit, std::memory_order_release);
        return e;
    }
};

// Number of SMs of the current device, queried once per device.
inline int sm_count() {
    static std::atomic<int> cache[kMaxDevices];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 1;
    const bool cacheable = dev >= 0 && dev < kMaxDevices;
    if (cacheable) {
        if (const int n = cache[dev].load(std::memory_order_relaxed); n > 0) return n;
    }
    int n = 0;
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) return 1;
    if (cacheable) cache[dev].store(n, std::memory_order_relaxed);
    return n;
}

// ------------------------------------------------------------ bf16 helpers

__device__ __forceinline__ float bf16lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf16hi(uint32_t v) { return __uint_as_float(v & 0xffff0000u); }

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);  // .x = lo, .y = hi, RNE
    return *reinterpret_cast<uint32_t*>(&h);
}

// Eight consecutive activation elements starting at p (16-byte aligned for
// bf16, 32-byte aligned for fp32) widened to fp32.
template <typename TA>
struct Vec8;

template <>
struct Vec8<__nv_bfloat16> {
    __device__ __forceinline__ static void load(const __nv_bfloat16* p, float (&v)[8]) {
        uint4 u = *reinterpret_cast<const uint4*>(p);
        v[0] = bf16lo(u.x); v[1] = bf16hi(u.x); v[2] = bf16lo(u.y); v[3] = bf16hi(u.y);
        v[4] = bf16lo(u.z); v[5] = bf16hi(u.z); v[6] = bf16lo(u.w); v[7] = bf16hi(u.w);
    }
    __device__ __forceinline__ static void store(__nv_bfloat16* p, const float (&v)[8]) {
        uint4 u;
        u.x = pack_bf16x2(v[0], v[1]); u.y = pack_bf16x2(v[2], v[3]);
        u.z = pack_bf16x2(v[4], v[5]); u.w = pack_bf16x2(v[6], v[7]);
        *reinterpret_cast<uint4*>(p) = u;
    }
};

template <>
struct Vec8<float> {
    __device__ __forceinline__ static void load(const float* p, float (&v)[8]) {
        float4 a = *reinterpret_cast<const float4*>(p);
        float4 b = *reinterpret_cast<const float4*>(p + 4);
        v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
    }
    __device__ __forceinline__ static void store(float* p, const float (&v)[8]) {
        *reinterpret_cast<float4*>(p) = make_float4(v[0], v[1], v[2], v[3]);
        *reinterpret_cast<float4*>(p + 4) = make_float4(v[4], v[5], v[6], v[7]);
    }
};

template <typename T>
__device__ __forceinline__ float to_f32(T v);
template <>
__device__ __forceinline__ float to_f32<float>(float v) { return v; }
template <>
__device__ __forceinline__ float to_f32<__nv_bfloat16>(__nv_bfloat16 v) { return __bfloat162float(v); }

template <typename T>
__device__ __forceinline__ T from_f32(float v);
template <>
__device__ __forceinline__ float from_f32<float>(float v) { return v; }
template <>
__device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float v) { return __float2bfloat16_rn(v); }

// 16-byte load of data read once (expert weights): not kept in L1.
__device__ __forceinline__ uint4 ld_stream16(const void* p) {
    uint4 r;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
                 : "l"(p));
    return r;
}

// ------------------------------------------------------- weight decoding

// e4m3 byte -> fp32 value (sign, 4-bit exponent with bias 7, 3-bit mantissa,
// subnormals at exponent 0; the NaN code is never produced by a quantiser).
__device__ __forceinline__ float e4m3_to_f32(uint32_t b) {
    uint32_t sign = (b & 0x80u) << 24;
    uint32_t em = b & 0x7fu;
    float mag;
    if (em >= 8u) {
        // normal: rebias exponent 7 -> 127, mantissa 3 -> 23 bits
        mag = __uint_as_float(((em >> 3) + 120u) << 23 | (em & 7u) << 20);
    } else {
        mag = (float)em * 0.001953125f;  // m * 2^-9
    }
    return __uint_as_float(__float_as_uint(mag) | sign);
}

// two e4m3 values (low byte = first element) -> two fp32, through the
// hardware e4m3x2 -> f16x2 conversion (every e4m3 value is exact in f16)
__device__ __forceinline__ float2 e4m3x2_to_f32x2(uint32_t two_bytes) {
    uint32_t h2;
    asm("cvt.rn.f16x2.e4m3x2 %0, %1;" : "=r"(h2) : "h"((unsigned short)two_bytes));
    __half2 h = *reinterpret_cast<__half2*>(&h2);
    return __half22float2(h);
}

// signed 4-bit value of nibble n (two's complement)
__device__ __forceinline__ float int4_to_f32(uint32_t n) { return (float)((int32_t)(n << 28) >> 28); }

// FP4 E2M1 code (sign in bit 3, exponent bits 2-1 with bias 1, mantissa bit
// 0) -> fp32, exact: the exponent and mantissa bits land in the fp32
// exponent field 0..3 and the top mantissa bit, which reads as the value
// times 2^-126 (the E2M1 subnormal 0.5 as the fp32 subnormal 2^-127), then
// one multiply by 2^126.
__device__ __forceinline__ float e2m1_to_f32(uint32_t c) {
    const float v = __uint_as_float(((c & 8u) << 28) | ((c & 7u) << 22));
    return v * __uint_as_float(0x7e800000u);  // 2^126
}

// E8M0 scale byte s -> 2^(s - 127) (s = 0: the fp32 subnormal 2^-127; 255: NaN)
__device__ __forceinline__ float e8m0_to_f32(uint32_t s) {
    return s == 255u ? __uint_as_float(0x7fc00000u) : s ? __uint_as_float(s << 23) : __uint_as_float(0x00400000u);
}

// ------------------------------------------------------------- silu

__device__ __forceinline__ float silu_mul(float g, float u) { return g / (1.0f + expf(-g)) * u; }

// ------------------------------------------------------------ errors

constexpr int32_t kErrTimeout = 1;

__device__ __forceinline__ void set_error(int32_t* err, int32_t code) {
    if (err) atomicOr(err, code);
}

}  // namespace gbmoe
