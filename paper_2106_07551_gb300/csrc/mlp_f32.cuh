// fp32 MLP forward on CUDA cores for a block of policy rows (one row = one
// observation whose acting agent's policy produces 3..5 logits).
//
// logits = W3 relu(W2 relu(W1 x + b1) + b2) + b3, weights resident in shared
// memory in the F32Layout (k-major W1, W2). The 256 threads of a CTA tile a
// pass of rows x H outputs as TY row-groups of 4 rows times TX column-groups of
// 8 columns (columns {4tx..4tx+3} and {H/2+4tx..}); each k step then costs one
// 16-byte load of the 4 rows' inputs (amortised over 4 k) and two 16-byte
// weight loads for 32 FMAs. A 16-byte shared load is served per half-warp, one
// 128-byte wavefront per 128 distinct bytes, so lanes are laid out to give
// every half-warp 8 column groups x 2 row groups: a weight load then costs 2
// wavefronts per warp and an input load 2 (16 column groups in a half-warp
// would cost 4 per weight load). Every row-group may use its own policy (the caller
// passes that group's weight pointer), so rows compacted by acting policy in
// multiples of 4 need no further sorting. Layer 3 is folded into layer 2's
// epilogue: per-thread partial dot products reduced across the TX lanes of the
// row-group with warp shuffles.
#pragma once

#include "internal.h"

namespace malib {

template <int IN, int H, int A>
struct MlpF32 {
    using L = F32Layout<IN, H, A>;
    static constexpr int kThreads = 256;
    static constexpr int TX = H / 8;
    static constexpr int TY = kThreads / TX;
    static constexpr int kRowsPerPass = TY * 4;
    static constexpr int XS = (IN + 3) / 4 * 4;   // input row stride (floats)
    static constexpr int HS = H + 4;              // hidden row stride (bank-skewed)
    static constexpr int LS = (A + 3) / 4 * 4;    // logits row stride
    static constexpr int TYW = 32 / TX;           // row-groups per warp
    static_assert(TX == 8 || TX == 16, "8 or 16 column groups (H = 64 or 128)");
    static_assert(A <= 8, "at most 8 actions");

    // Lane -> (column group, row group). TX 16: lanes 0-7 and 8-15 hold column
    // groups 0-7 of row groups 2w and 2w+1, lanes 16-31 column groups 8-15.
    // TX 8: lanes 8r..8r+7 hold column groups 0-7 of row group 4w+r.
    __device__ static int col_group() {
        const int lane = threadIdx.x & 31;
        return TX == 16 ? ((lane & 7) | ((lane >> 4) << 3)) : (lane & 7);
    }
    __device__ static int row_group() {
        const int lane = threadIdx.x & 31;
        const int tyl = TX == 16 ? ((lane >> 3) & 1) : (lane >> 3);
        return (threadIdx.x >> 5) * TYW + tyl;
    }

    // First local row of the warp's first row-group (for warp-uniform skips).
    __device__ static int warp_first_row() { return (threadIdx.x >> 5) * TYW * 4; }

    // One pass: rows [row0, row0 + kRowsPerPass) of X -> the same rows of LG.
    // w: weight blob of the calling thread's row-group. `active` must be
    // uniform across the warp. Contains two __syncthreads (all threads call).
    __device__ static void pass(const float* __restrict__ X, float* __restrict__ H1,
                                float* __restrict__ LG, const float* __restrict__ w, int row0,
                                bool active) {
        const int tx = col_group();
        const int ty = row_group();
        const int lr = ty * 4;
        const int c0 = tx * 4, c1 = H / 2 + tx * 4;
        float acc[4][8];

        if (active) {
            const float4 bA = *reinterpret_cast<const float4*>(w + L::kB1 + c0);
            const float4 bB = *reinterpret_cast<const float4*>(w + L::kB1 + c1);
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                acc[i][0] = bA.x; acc[i][1] = bA.y; acc[i][2] = bA.z; acc[i][3] = bA.w;
                acc[i][4] = bB.x; acc[i][5] = bB.y; acc[i][6] = bB.z; acc[i][7] = bB.w;
            }
            const float* xr = X + (size_t)(row0 + lr) * XS;
#pragma unroll
            for (int k0 = 0; k0 < IN; k0 += 4) {
                float4 xa[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) xa[i] = *reinterpret_cast<const float4*>(xr + i * XS + k0);
#pragma unroll
                for (int kk = 0; kk < 4; ++kk) {
                    if (k0 + kk < IN) {
                        const float* wk = w + L::kW1T + (k0 + kk) * H;
                        const float4 wA = *reinterpret_cast<const float4*>(wk + c0);
                        const float4 wB = *reinterpret_cast<const float4*>(wk + c1);
#pragma unroll
                        for (int i = 0; i < 4; ++i) {
                            const float xv = kk == 0 ? xa[i].x : kk == 1 ? xa[i].y : kk == 2 ? xa[i].z : xa[i].w;
                            acc[i][0] = fmaf(xv, wA.x, acc[i][0]);
                            acc[i][1] = fmaf(xv, wA.y, acc[i][1]);
                            acc[i][2] = fmaf(xv, wA.z, acc[i][2]);
                            acc[i][3] = fmaf(xv, wA.w, acc[i][3]);
                            acc[i][4] = fmaf(xv, wB.x, acc[i][4]);
                            acc[i][5] = fmaf(xv, wB.y, acc[i][5]);
                            acc[i][6] = fmaf(xv, wB.z, acc[i][6]);
                            acc[i][7] = fmaf(xv, wB.w, acc[i][7]);
                        }
                    }
                }
            }
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                float4 hA = make_float4(fmaxf(acc[i][0], 0.f), fmaxf(acc[i][1], 0.f),
                                        fmaxf(acc[i][2], 0.f), fmaxf(acc[i][3], 0.f));
                float4 hB = make_float4(fmaxf(acc[i][4], 0.f), fmaxf(acc[i][5], 0.f),
                                        fmaxf(acc[i][6], 0.f), fmaxf(acc[i][7], 0.f));
                *reinterpret_cast<float4*>(H1 + (lr + i) * HS + c0) = hA;
                *reinterpret_cast<float4*>(H1 + (lr + i) * HS + c1) = hB;
            }
        }
        __syncthreads();

        if (active) {
            const float4 bA = *reinterpret_cast<const float4*>(w + L::kB2 + c0);
            const float4 bB = *reinterpret_cast<const float4*>(w + L::kB2 + c1);
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                acc[i][0] = bA.x; acc[i][1] = bA.y; acc[i][2] = bA.z; acc[i][3] = bA.w;
                acc[i][4] = bB.x; acc[i][5] = bB.y; acc[i][6] = bB.z; acc[i][7] = bB.w;
            }
            const float* hr = H1 + lr * HS;
#pragma unroll 2
            for (int k0 = 0; k0 < H; k0 += 4) {
                float4 ha[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) ha[i] = *reinterpret_cast<const float4*>(hr + i * HS + k0);
#pragma unroll
                for (int kk = 0; kk < 4; ++kk) {
                    const float* wk = w + L::kW2T + (k0 + kk) * H;
                    const float4 wA = *reinterpret_cast<const float4*>(wk + c0);
                    const float4 wB = *reinterpret_cast<const float4*>(wk + c1);
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        const float hv = kk == 0 ? ha[i].x : kk == 1 ? ha[i].y : kk == 2 ? ha[i].z : ha[i].w;
                        acc[i][0] = fmaf(hv, wA.x, acc[i][0]);
                        acc[i][1] = fmaf(hv, wA.y, acc[i][1]);
                        acc[i][2] = fmaf(hv, wA.z, acc[i][2]);
                        acc[i][3] = fmaf(hv, wA.w, acc[i][3]);
                        acc[i][4] = fmaf(hv, wB.x, acc[i][4]);
                        acc[i][5] = fmaf(hv, wB.y, acc[i][5]);
                        acc[i][6] = fmaf(hv, wB.z, acc[i][6]);
                        acc[i][7] = fmaf(hv, wB.w, acc[i][7]);
                    }
                }
            }
            // layer 3 partials over this thread's 8 columns
            float pl[4][A];
#pragma unroll
            for (int a = 0; a < A; ++a) {
                const float4 vA = *reinterpret_cast<const float4*>(w + L::kW3 + a * H + c0);
                const float4 vB = *reinterpret_cast<const float4*>(w + L::kW3 + a * H + c1);
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    float s = fmaxf(acc[i][0], 0.f) * vA.x;
                    s = fmaf(fmaxf(acc[i][1], 0.f), vA.y, s);
                    s = fmaf(fmaxf(acc[i][2], 0.f), vA.z, s);
                    s = fmaf(fmaxf(acc[i][3], 0.f), vA.w, s);
                    s = fmaf(fmaxf(acc[i][4], 0.f), vB.x, s);
                    s = fmaf(fmaxf(acc[i][5], 0.f), vB.y, s);
                    s = fmaf(fmaxf(acc[i][6], 0.f), vB.z, s);
                    s = fmaf(fmaxf(acc[i][7], 0.f), vB.w, s);
                    pl[i][a] = s;
                }
            }
            // reduce over the lanes of the row-group: tx bits are lane bits
            // 0-2 (and lane bit 4 when TX = 16)
#pragma unroll
            for (int o = 1; o <= (TX == 16 ? 16 : 4); o <<= 1) {
                if (o == 8) continue;
#pragma unroll
                for (int i = 0; i < 4; ++i)
#pragma unroll
                    for (int a = 0; a < A; ++a) pl[i][a] += __shfl_xor_sync(0xffffffffu, pl[i][a], o);
            }
            if (tx == 0) {
#pragma unroll
                for (int i = 0; i < 4; ++i)
#pragma unroll
                    for (int a = 0; a < A; ++a) LG[(row0 + lr + i) * LS + a] = pl[i][a] + w[L::kB3 + a];
            }
        }
        __syncthreads();
    }
};

}  // namespace malib
