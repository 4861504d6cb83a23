// Layout of the grouped-FFN work lists (see ffn_sched.cu).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace gbmoe {

constexpr int kSchedHeader = 8;  // [0] active experts, [1] tiles, rest reserved
constexpr int kSchedMinBM = 32;  // smallest tile height any FFN route uses

inline int64_t sched_max_tiles(int E, int64_t n_rows, int BM) { return (n_rows + BM - 1) / BM + E; }

// int offset of the int2 tile list (8-byte aligned)
__host__ __device__ inline size_t sched_tiles_offset(int E) {
    size_t o = (size_t)kSchedHeader + E + (E + 1);
    return (o + 1) & ~(size_t)1;
}

cudaError_t launch_ffn_schedule(const int32_t* counts, int E, int64_t n_rows, int BM, int32_t* sched,
                                cudaStream_t stream);

}  // namespace gbmoe
