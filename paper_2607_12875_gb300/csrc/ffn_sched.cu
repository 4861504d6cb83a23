// Work lists for the grouped expert FFN, built on the device from the
// per-expert counts (the host never learns them, so nothing synchronises):
// the ascending list of experts that received rows, and the list of
// BM-row tiles (expert, tile index inside the expert) in expert order.
#include "common.cuh"
#include "ffn_sched.h"

namespace gbmoe {

size_t ffn_sched_ints(int E, int64_t n_rows) {
    return (size_t)kSchedHeader + E + (E + 1) + 2 * (size_t)sched_max_tiles(E, n_rows, kSchedMinBM) + 64;
}

__global__ void __launch_bounds__(512)
ffn_schedule_kernel(const int32_t* __restrict__ counts, int E, int64_t n_rows, int BM, int32_t* __restrict__ sched) {
    pdl_enter();
    __shared__ int32_t s_warp_t[16], s_warp_a[16];
    const int e = threadIdx.x, lane = e & 31, warp = e >> 5;
    int cnt = 0;
    if (e < E) cnt = counts ? counts[e] : (int)n_rows;
    const int nt = (cnt + BM - 1) / BM;
    const int act = cnt > 0 ? 1 : 0;
    int it = nt, ia = act;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
        int ot = __shfl_up_sync(0xffffffffu, it, d), oa = __shfl_up_sync(0xffffffffu, ia, d);
        if (lane >= d) { it += ot; ia += oa; }
    }
    if (lane == 31) { s_warp_t[warp] = it; s_warp_a[warp] = ia; }
    __syncthreads();
    if (warp == 0) {
        const int nw = blockDim.x >> 5;
        int wt = lane < nw ? s_warp_t[lane] : 0, wa = lane < nw ? s_warp_a[lane] : 0;
        int st = wt, sa = wa;
#pragma unroll
        for (int d = 1; d < 32; d <<= 1) {
            int ot = __shfl_up_sync(0xffffffffu, st, d), oa = __shfl_up_sync(0xffffffffu, sa, d);
            if (lane >= d) { st += ot; sa += oa; }
        }
        if (lane < nw) { s_warp_t[lane] = st - wt; s_warp_a[lane] = sa - wa; }
        if (lane == nw - 1) { sched[0] = sa; sched[1] = st; }
    }
    __syncthreads();
    const int tile0 = s_warp_t[warp] + it - nt;
    const int aidx = s_warp_a[warp] + ia - act;
    if (e < E) {
        int32_t* active = sched + kSchedHeader;
        int32_t* tile_off = active + E;
        int2* tiles = reinterpret_cast<int2*>(sched + sched_tiles_offset(E));
        if (act) active[aidx] = e;
        tile_off[e] = tile0;
        if (e == E - 1) tile_off[E] = tile0 + nt;
        for (int m = 0; m < nt; ++m) tiles[tile0 + m] = make_int2(e, m);
    }
}

cudaError_t launch_ffn_schedule(const int32_t* counts, int E, int64_t n_rows, int BM, int32_t* sched,
                                cudaStream_t stream) {
    if (const cudaError_t le = launch_k(ffn_schedule_kernel, dim3(1), dim3(512), 0, stream, counts, E, n_rows, BM,
            sched); le != cudaSuccess)
        return le;
    return cudaGetLastError();
}

}  // namespace gbmoe
