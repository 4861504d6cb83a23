// Fused MoE, grouping step: stable counting sort of the (token, slot) pairs
// by expert. Three small kernels: per-block histograms, one scan that turns
// them into counts, offsets and per-block bases, and a scatter that ranks
// pairs inside a block in pair order (warp match + warp-ordered running
// counters), so the result is the stable order whatever the scheduling.
// Up to 1024 pairs (decode) all three steps run in one CTA. A pair whose
// expert id is outside [0, E) is dropped: pair_pos[p] = -1, and the sorted
// positions past the last kept pair hold -1.
#include "common.cuh"
#include "kernels.h"

namespace gbmoe {

constexpr int kPermBlock = 1024;  // pairs per block (one per thread)

int permute_blocks(int64_t P) { return (int)((P + kPermBlock - 1) / kPermBlock); }

// block histograms [nblk][E] + per-block bases [nblk][E]
size_t permute_scratch_ints(int64_t P, int E) { return 2 * (size_t)permute_blocks(P) * E; }

__global__ void __launch_bounds__(kPermBlock)
perm_hist_kernel(const int32_t* __restrict__ ids, int64_t P, int E, int32_t* __restrict__ block_hist) {
    pdl_enter();
    extern __shared__ int32_t s_hist[];
    for (int e = threadIdx.x; e < E; e += blockDim.x) s_hist[e] = 0;
    __syncthreads();
    int64_t p = (int64_t)blockIdx.x * kPermBlock + threadIdx.x;
    if (p < P) {
        const int e = ids[p];
        if (e >= 0 && e < E) atomicAdd(&s_hist[e], 1);  // out-of-range ids are dropped
    }
    __syncthreads();
    for (int e = threadIdx.x; e < E; e += blockDim.x) block_hist[(size_t)blockIdx.x * E + e] = s_hist[e];
}

// One block, thread e owns expert e: walks the block histograms in order.
__global__ void __launch_bounds__(512)
perm_scan_kernel(const int32_t* __restrict__ block_hist, int nblk, int E, int32_t* __restrict__ counts,
                 int32_t* __restrict__ offsets, int32_t* __restrict__ block_base) {
    pdl_enter();
    __shared__ int32_t s_warp[16];
    const int e = threadIdx.x;
    int run = 0;
    if (e < E)
        for (int b = 0; b < nblk; ++b) {
            block_base[(size_t)b * E + e] = run;
            run += block_hist[(size_t)b * E + e];
        }
    // exclusive scan of the counts over experts
    const int lane = e & 31, warp = e >> 5;
    int v = (e < E) ? run : 0, incl = v;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
        int o = __shfl_up_sync(0xffffffffu, incl, d);
        if (lane >= d) incl += o;
    }
    if (lane == 31) s_warp[warp] = incl;
    __syncthreads();
    if (warp == 0) {
        int w = (lane < (int)(blockDim.x >> 5)) ? s_warp[lane] : 0, wi = w;
#pragma unroll
        for (int d = 1; d < 32; d <<= 1) {
            int o = __shfl_up_sync(0xffffffffu, wi, d);
            if (lane >= d) wi += o;
        }
        if (lane < 16) s_warp[lane] = wi - w;  // exclusive warp prefix
    }
    __syncthreads();
    int excl = s_warp[warp] + incl - v;
    if (e < E) {
        counts[e] = run;
        offsets[e] = excl;
        if (e == E - 1) offsets[E] = excl + run;
        for (int b = 0; b < nblk; ++b) block_base[(size_t)b * E + e] += excl;
    }
}

__global__ void __launch_bounds__(kPermBlock)
perm_scatter_kernel(const int32_t* __restrict__ ids, int64_t P, int E, const int32_t* __restrict__ block_base,
                    const int32_t* __restrict__ offsets, int32_t* __restrict__ sorted_pair,
                    int32_t* __restrict__ pair_pos) {
    pdl_enter();
    extern __shared__ int32_t s_run[];
    for (int e = threadIdx.x; e < E; e += blockDim.x) s_run[e] = block_base[(size_t)blockIdx.x * E + e];
    __syncthreads();
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t p = (int64_t)blockIdx.x * kPermBlock + threadIdx.x;
    const int id = p < P ? ids[p] : -1;
    const bool valid = id >= 0 && id < E;
    const int e = valid ? id : -1 - lane;  // invalid lanes never match a real expert
    const uint32_t peers = __match_any_sync(0xffffffffu, e);
    const int rank = __popc(peers & ((1u << lane) - 1u));
    const bool leader = rank == 0;
    int pos = 0;
    // warps take their places in pair order
    for (int w = 0; w < kPermBlock / 32; ++w) {
        if (warp == w && valid) {
            pos = s_run[e] + rank;
            __syncwarp(peers);
            if (leader) s_run[e] += __popc(peers);
        }
        __syncthreads();
    }
    if (valid) {
        sorted_pair[pos] = (int32_t)p;
        pair_pos[p] = pos;
    } else if (p < P) {
        pair_pos[p] = -1;  // dropped pair: no slot
    }
    // positions past the last kept pair (only when pairs were dropped) hold -1
    if (p < P && p >= offsets[E]) sorted_pair[p] = -1;
}

// P <= kPermBlock: histogram, scan and stable scatter in one CTA (one pair
// per thread). Same order and outputs as the three kernels above with one
// block: the block base of expert e is its offset.
__global__ void __launch_bounds__(kPermBlock)
perm_small_kernel(const int32_t* __restrict__ ids, int64_t P, int E, int32_t* __restrict__ counts,
                  int32_t* __restrict__ offsets, int32_t* __restrict__ sorted_pair, int32_t* __restrict__ pair_pos) {
    pdl_enter();
    extern __shared__ int32_t s_run[];  // [E]: histogram, then running positions
    __shared__ int32_t s_warp[kPermBlock / 32];
    __shared__ int32_t s_kept;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int e = threadIdx.x; e < E; e += blockDim.x) s_run[e] = 0;
    __syncthreads();
    const int p = threadIdx.x;
    const int id = p < P ? ids[p] : -1;
    const bool valid = id >= 0 && id < E;  // out-of-range ids are dropped
    if (valid) atomicAdd(&s_run[id], 1);
    __syncthreads();
    // exclusive scan of the counts over experts (thread e owns expert e; E <= 512)
    const int cnt = threadIdx.x < E ? s_run[threadIdx.x] : 0;
    int incl = cnt;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
        int o = __shfl_up_sync(0xffffffffu, incl, d);
        if (lane >= d) incl += o;
    }
    if (lane == 31) s_warp[warp] = incl;
    __syncthreads();
    if (warp == 0) {
        int w = s_warp[lane], wi = w;
#pragma unroll
        for (int d = 1; d < 32; d <<= 1) {
            int o = __shfl_up_sync(0xffffffffu, wi, d);
            if (lane >= d) wi += o;
        }
        s_warp[lane] = wi - w;  // exclusive warp prefix
    }
    __syncthreads();
    const int excl = s_warp[warp] + incl - cnt;
    if (threadIdx.x < E) {
        counts[threadIdx.x] = cnt;
        offsets[threadIdx.x] = excl;
        if (threadIdx.x == E - 1) {
            offsets[E] = excl + cnt;
            s_kept = excl + cnt;
        }
        s_run[threadIdx.x] = excl;
    }
    __syncthreads();
    // stable scatter: warps take their places in pair order
    const int e = valid ? id : -1 - lane;  // invalid lanes never match a real expert
    const uint32_t peers = __match_any_sync(0xffffffffu, e);
    const int rank = __popc(peers & ((1u << lane) - 1u));
    int pos = 0;
    for (int w = 0; w < kPermBlock / 32; ++w) {
        if (warp == w && valid) {
            pos = s_run[e] + rank;
            __syncwarp(peers);
            if (rank == 0) s_run[e] += __popc(peers);
        }
        __syncthreads();
    }
    if (valid) {
        sorted_pair[pos] = p;
        pair_pos[p] = pos;
    } else if (p < P) {
        pair_pos[p] = -1;  // dropped pair: no slot
    }
    if (p < P && p >= s_kept) sorted_pair[p] = -1;  // past the last kept pair
}

cudaError_t launch_permute(const int32_t* topk_ids, int64_t P, int E, int32_t* counts, int32_t* offsets,
                           int32_t* sorted_pair, int32_t* pair_pos, int32_t* scratch, cudaStream_t stream) {
    const int nblk = permute_blocks(P);
    if (nblk == 1)
        return launch_k(perm_small_kernel, dim3(1), dim3(kPermBlock), E * sizeof(int32_t), stream, topk_ids, P, E,
                        counts, offsets, sorted_pair, pair_pos);
    int32_t* block_hist = scratch;
    int32_t* block_base = scratch + (size_t)nblk * E;
    if (nblk > 0) {
        if (const cudaError_t le = launch_k(perm_hist_kernel, dim3(nblk), dim3(kPermBlock), E * sizeof(int32_t),
                stream, topk_ids, P, E, block_hist); le != cudaSuccess)
            return le;
        cudaError_t err = cudaGetLastError();
        if (err != cudaSuccess) return err;
    }
    if (const cudaError_t le = launch_k(perm_scan_kernel, dim3(1), dim3(512), 0, stream, block_hist, nblk, E,
            counts, offsets, block_base); le != cudaSuccess)
        return le;
    cudaError_t err = cudaGetLastError();
    if (err != cudaSuccess || nblk == 0) return err;
    if (const cudaError_t le = launch_k(perm_scatter_kernel, dim3(nblk), dim3(kPermBlock), E * sizeof(int32_t),
            stream, topk_ids, P, E, block_base, offsets, sorted_pair, pair_pos); le != cudaSuccess)
        return le;
    return cudaGetLastError();
}

}  // namespace gbmoe
