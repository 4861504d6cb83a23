// moe_permute_noalloc: the grouping step with its scratch in a static device
// array instead of a caller-provided workspace.
//
// Some callers cannot allocate device memory for the call: plain C hosts
// that link this library without any allocator of their own, engines that
// reserve all device memory up front and hand out no extra buffers, or code
// running where cudaMalloc is not allowed. For them the permutation keeps
// its block histograms and block bases in the file-scope array below, which
// every GPU that loads the library holds until the process exits.
//
// The array's name, used in host code, is only a host-side stand-in, not a
// device address. Its device address is looked up once per device, with
// that device current, by cudaGetSymbolAddress; the first call on each
// device does this and should therefore come before any stream capture.
// The address is kept until the process exits: a reset of the device's
// context (cudaDeviceReset) would leave it stale, so the call is not for
// processes that reset a device and go on.
// All calls share the array and it keeps the previous call's contents, so
// two calls that overlap on the GPU (different streams, no ordering) race.
// The scan and scatter overwrite every entry they read, so nothing needs
// clearing between calls.
#include <mutex>

#include "common.cuh"
#include "kernels.h"

namespace {

constexpr size_t kStaticScratchInts = 262144;  // 1 MiB

static __device__ __align__(256) int32_t g_permute_scratch[kStaticScratchInts];

constexpr int kMaxDevices = 64;
std::mutex g_mutex;
int32_t* g_scratch_ptr[kMaxDevices] = {};

// Device address of the static scratch on the current device, or null.
int32_t* scratch_on_current_device(cudaError_t* err) {
    int dev = -1;
    *err = cudaGetDevice(&dev);
    if (*err != cudaSuccess) return nullptr;
    if (dev < 0 || dev >= kMaxDevices) {
        *err = cudaErrorInvalidDevice;
        return nullptr;
    }
    std::lock_guard<std::mutex> lock(g_mutex);
    if (!g_scratch_ptr[dev]) {
        void* p = nullptr;
        *err = cudaGetSymbolAddress(&p, g_permute_scratch);
        if (*err != cudaSuccess) return nullptr;
        g_scratch_ptr[dev] = static_cast<int32_t*>(p);
    }
    return g_scratch_ptr[dev];
}

}  // namespace

extern "C" int moe_permute_noalloc(const gbmoe_config* cfg, const int32_t* topk_ids, int32_t* counts,
                                   int32_t* offsets, int32_t* sorted_pair, int32_t* pair_pos, void* stream) {
    int s = gbmoe_check_config(cfg);
    if (s) return s;
    if (!topk_ids || !counts || !offsets || !sorted_pair || !pair_pos) return GBMOE_EINVAL;
    auto al4 = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 3u) == 0; };
    if (!al4(topk_ids) || !al4(counts) || !al4(offsets) || !al4(sorted_pair) || !al4(pair_pos)) return GBMOE_EINVAL;
    const int64_t P = (int64_t)cfg->T * cfg->top_k;
    if (gbmoe::permute_scratch_ints(P, cfg->E) > kStaticScratchInts) return GBMOE_EUNSUPPORTED;
    cudaError_t err;
    int32_t* scratch = scratch_on_current_device(&err);
    if (!scratch) return GBMOE_ECUDA;
    err = gbmoe::launch_permute(topk_ids, P, cfg->E, counts, offsets, sorted_pair, pair_pos, scratch,
                                static_cast<cudaStream_t>(stream));
    return err == cudaSuccess ? GBMOE_OK : GBMOE_ECUDA;
}
