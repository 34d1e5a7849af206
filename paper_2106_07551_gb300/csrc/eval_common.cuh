// Payoff-table helpers shared by the evaluation kernels: the block-level
// reduction of integer payoff sums and the validation of a pair of policy ids.
#pragma once

#include "device_common.cuh"
#include "internal.h"

namespace malib {

// Adds the block's payoff sums (sum r, sum r^2) into the pair's two 64-bit
// accumulators and its decision count into the call's total.
__device__ __forceinline__ void block_add_sums(long long s1, long long s2, long long nd,
                                               unsigned long long* acc2,
                                               unsigned long long* n_dec) {
    __shared__ long long red[3][32];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    s1 = warp_sum_ll(s1);
    s2 = warp_sum_ll(s2);
    nd = warp_sum_ll(nd);
    if (lane == 0) { red[0][warp] = s1; red[1][warp] = s2; red[2][warp] = nd; }
    __syncthreads();
    if (threadIdx.x == 0) {
        long long t1 = 0, t2 = 0, t3 = 0;
        for (int w = 0; w < (int)(blockDim.x + 31) / 32; ++w) {
            t1 += red[0][w]; t2 += red[1][w]; t3 += red[2][w];
        }
        atomicAdd(acc2, (unsigned long long)t1);
        atomicAdd(acc2 + 1, (unsigned long long)t2);
        atomicAdd(n_dec, (unsigned long long)t3);
    }
    __syncthreads();
}

__device__ __forceinline__ bool pair_ok(const EvalArgs& a, int p0, int p1) {
    if (p0 < 0 || p0 >= a.n_pol || p1 < 0 || p1 >= a.n_pol) return false;
    const int s0 = a.pol_seat[p0], s1 = a.pol_seat[p1];
    return (s0 == 0 || s0 == -1) && (s1 == 1 || s1 == -1);
}

}  // namespace malib
