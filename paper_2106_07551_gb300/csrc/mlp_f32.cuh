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

// Packed fp32 pair helpers: fma.rn.f32x2 performs two independent IEEE fp32
// fused multiply-adds (round to nearest), so results equal scalar fmaf.
__device__ __forceinline__ unsigned long long f2_dup(float v) {
    unsigned long long r;
    asm("mov.b64 %0, {%1, %1};" : "=l"(r) : "f"(v));
    return r;
}
__device__ __forceinline__ void f2_fma(unsigned long long& d, unsigned long long a,
                                       unsigned long long b) {
    asm("fma.rn.f32x2 %0, %1, %2, %0;" : "+l"(d) : "l"(a), "l"(b));
}
__device__ __forceinline__ float2 f2_split(unsigned long long v) {
    float lo, hi;
    asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
    return make_float2(lo, hi);
}
__device__ __forceinline__ unsigned long long f2_relu(unsigned long long v) {
    const float2 q = f2_split(v);
    unsigned long long r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(fmaxf(q.x, 0.f)), "f"(fmaxf(q.y, 0.f)));
    return r;
}

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
            // packed pairs: p[i][0..3] = column pairs (c0,c0+1) (c0+2,c0+3) (c1,..) (c1+2,..)
            unsigned long long p[4][4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                asm("mov.b64 %0, {%1, %2};" : "=l"(p[i][0]) : "f"(acc[i][0]), "f"(acc[i][1]));
                asm("mov.b64 %0, {%1, %2};" : "=l"(p[i][1]) : "f"(acc[i][2]), "f"(acc[i][3]));
                asm("mov.b64 %0, {%1, %2};" : "=l"(p[i][2]) : "f"(acc[i][4]), "f"(acc[i][5]));
                asm("mov.b64 %0, {%1, %2};" : "=l"(p[i][3]) : "f"(acc[i][6]), "f"(acc[i][7]));
            }
            const float* hr = H1 + lr * HS;
#pragma unroll 4
            for (int k0 = 0; k0 < H; k0 += 4) {
                float4 ha[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) ha[i] = *reinterpret_cast<const float4*>(hr + i * HS + k0);
#pragma unroll
                for (int kk = 0; kk < 4; ++kk) {
                    const float* wk = w + L::kW2T + (k0 + kk) * H;
                    const ulonglong2 wA = *reinterpret_cast<const ulonglong2*>(wk + c0);
                    const ulonglong2 wB = *reinterpret_cast<const ulonglong2*>(wk + c1);
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        const float hv = kk == 0 ? ha[i].x : kk == 1 ? ha[i].y : kk == 2 ? ha[i].z : ha[i].w;
                        const unsigned long long h2 = f2_dup(hv);
                        f2_fma(p[i][0], h2, wA.x);
                        f2_fma(p[i][1], h2, wA.y);
                        f2_fma(p[i][2], h2, wB.x);
                        f2_fma(p[i][3], h2, wB.y);
                    }
                }
            }
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const float2 q0 = f2_split(p[i][0]), q1 = f2_split(p[i][1]);
                const float2 q2 = f2_split(p[i][2]), q3 = f2_split(p[i][3]);
                acc[i][0] = q0.x; acc[i][1] = q0.y; acc[i][2] = q1.x; acc[i][3] = q1.y;
                acc[i][4] = q2.x; acc[i][5] = q2.y; acc[i][6] = q3.x; acc[i][7] = q3.y;
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


// 128-row pass of one policy with 8x8 register tiles (256 threads, H = 128):
// thread (tx, ty) computes rows ty + 16 i (i = 0..7) and columns
// {4tx..4tx+3} and {64+4tx..64+4tx+3}, accumulating adjacent column pairs
// with packed fp32 FMAs (2 FMAs per instruction). Per k it issues 4 16-byte
// shared loads (2 for its 8 inputs, amortised over 4 k, and 2 for its 8
// weights, which arrive as 4 column pairs), 8 duplications of an input into a
// pair, and 32 packed FMAs for 64 FMAs. Rows interleaved by 16 put the two row
// groups of a half-warp on adjacent rows, which the bank-skewed strides place
// in different banks. The weights arrive as separate pointers so that W2 can
// live in a buffer of its own (restaged per policy) while the small layers of
// several policies stay resident. Layer 3 is folded into layer 2's epilogue
// (shuffle reduction over the 16 column lanes of a row group, which share one
// warp). NI (1..8) is the number of 16-row blocks a pass computes: rows
// 0 .. 16 NI - 1, for passes whose compacted rows all lie there.
template <int IN, int A>
struct MlpF32T8 {
    static constexpr int H = 128;
    static constexpr int kThreads = 256;
    static constexpr int kRows = 128;
    static constexpr int XS = (IN + 3) / 4 * 4;
    static constexpr int HS = H + 4;
    static constexpr int LS = (A + 3) / 4 * 4;
    using u64 = unsigned long long;

    __device__ static int col_group() {
        const int lane = threadIdx.x & 31;
        return (lane & 7) | ((lane >> 4) << 3);
    }
    __device__ static int row_group() { return (threadIdx.x >> 5) * 2 + ((threadIdx.x >> 3) & 1); }

    // acc[i][p]: row i, column pair p (p 0,1: c0..c0+3; p 2,3: c1..c1+3)
    template <int NI>
    __device__ static void init(u64 (&acc)[8][4], const float* __restrict__ b, int c0, int c1) {
        const ulonglong2 bA = *reinterpret_cast<const ulonglong2*>(b + c0);
        const ulonglong2 bB = *reinterpret_cast<const ulonglong2*>(b + c1);
#pragma unroll
        for (int i = 0; i < NI; ++i) { acc[i][0] = bA.x; acc[i][1] = bA.y; acc[i][2] = bB.x; acc[i][3] = bB.y; }
    }

    // acc += rows' inputs [4 k from xa] x W rows k0..k0+3 (kk < kmax)
    template <int NI>
    __device__ static void block(u64 (&acc)[8][4], const float4 (&xa)[8], const float* __restrict__ W,
                                 int k0, int kmax, int c0, int c1) {
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {
            if (kk < kmax) {
                const ulonglong2 wA = *reinterpret_cast<const ulonglong2*>(W + (k0 + kk) * H + c0);
                const ulonglong2 wB = *reinterpret_cast<const ulonglong2*>(W + (k0 + kk) * H + c1);
                // all 8 duplications first, then the packed FMAs column pair by
                // column pair, so no FMA waits on the duplication just before it
                u64 x2[8];
#pragma unroll
                for (int i = 0; i < NI; ++i)
                    x2[i] = f2_dup(kk == 0 ? xa[i].x : kk == 1 ? xa[i].y : kk == 2 ? xa[i].z : xa[i].w);
#pragma unroll
                for (int i = 0; i < NI; ++i) f2_fma(acc[i][0], x2[i], wA.x);
#pragma unroll
                for (int i = 0; i < NI; ++i) f2_fma(acc[i][1], x2[i], wA.y);
#pragma unroll
                for (int i = 0; i < NI; ++i) f2_fma(acc[i][2], x2[i], wB.x);
#pragma unroll
                for (int i = 0; i < NI; ++i) f2_fma(acc[i][3], x2[i], wB.y);
            }
        }
    }

    // Layer 1 into H1 (rows of X [128][XS]). Ends with __syncthreads.
    template <int NI = 8>
    __device__ static void layer1(const float* __restrict__ X, float* __restrict__ H1,
                                  const float* __restrict__ W1T, const float* __restrict__ b1) {
        const int tx = col_group(), ty = row_group();
        const int c0 = tx * 4, c1 = H / 2 + tx * 4;
        u64 acc[8][4];
        init<NI>(acc, b1, c0, c1);
#pragma unroll
        for (int k0 = 0; k0 < IN; k0 += 4) {
            float4 xa[8];
#pragma unroll
            for (int i = 0; i < NI; ++i)
                xa[i] = *reinterpret_cast<const float4*>(X + (ty + 16 * i) * XS + k0);
            block<NI>(acc, xa, W1T, k0, IN - k0, c0, c1);
        }
#pragma unroll
        for (int i = 0; i < NI; ++i) {
            float* hr = H1 + (ty + 16 * i) * HS;
            const float2 p0 = f2_split(acc[i][0]), p1 = f2_split(acc[i][1]);
            const float2 p2 = f2_split(acc[i][2]), p3 = f2_split(acc[i][3]);
            *reinterpret_cast<float4*>(hr + c0) = make_float4(fmaxf(p0.x, 0.f), fmaxf(p0.y, 0.f),
                                                              fmaxf(p1.x, 0.f), fmaxf(p1.y, 0.f));
            *reinterpret_cast<float4*>(hr + c1) = make_float4(fmaxf(p2.x, 0.f), fmaxf(p2.y, 0.f),
                                                              fmaxf(p3.x, 0.f), fmaxf(p3.y, 0.f));
        }
        __syncthreads();
    }

    // Layers 2 and 3: H1 -> logits rows of LG [128][LS]. Ends with __syncthreads.
    template <int NI = 8>
    __device__ static void layer23(const float* __restrict__ H1, float* __restrict__ LG,
                                   const float* __restrict__ W2T, const float* __restrict__ b2,
                                   const float* __restrict__ W3, const float* __restrict__ b3) {
        const int tx = col_group(), ty = row_group();
        const int c0 = tx * 4, c1 = H / 2 + tx * 4;
        u64 acc[8][4];
        init<NI>(acc, b2, c0, c1);
#pragma unroll 2
        for (int k0 = 0; k0 < H; k0 += 4) {
            float4 ha[8];
#pragma unroll
            for (int i = 0; i < NI; ++i)
                ha[i] = *reinterpret_cast<const float4*>(H1 + (ty + 16 * i) * HS + k0);
            block<NI>(acc, ha, W2T, k0, 4, c0, c1);
        }
        // layer 3: ReLU once, then per row and action a packed dot product over
        // the thread's 4 column pairs and the sum of its two halves
        static_assert(A == 3, "the reduce-scatter below places 3 logits per row");
        static_assert(NI >= 1 && NI <= 8, "1 to 8 row blocks");
#pragma unroll
        for (int i = 0; i < NI; ++i)
#pragma unroll
            for (int p = 0; p < 4; ++p) acc[i][p] = f2_relu(acc[i][p]);
        // the reduce-scatter runs on 8 (NI > 4) or 4 row blocks; blocks beyond
        // NI enter it as zeros and their rows hold no hand
        constexpr int NR = NI > 4 ? 8 : 4;
        constexpr int V = NR * A;                 // partial logits of this thread
        float v0[V];
#pragma unroll
        for (int j = NI * A; j < V; ++j) v0[j] = 0.f;
#pragma unroll
        for (int a = 0; a < A; ++a) {
            const ulonglong2 wA = *reinterpret_cast<const ulonglong2*>(W3 + a * H + c0);
            const ulonglong2 wB = *reinterpret_cast<const ulonglong2*>(W3 + a * H + c1);
#pragma unroll
            for (int i = 0; i < NI; ++i) {
                u64 t = 0ull;
                f2_fma(t, acc[i][0], wA.x);
                f2_fma(t, acc[i][1], wA.y);
                f2_fma(t, acc[i][2], wB.x);
                f2_fma(t, acc[i][3], wB.y);
                const float2 q = f2_split(t);
                v0[i * A + a] = q.x + q.y;
            }
        }
        // Reduce-scatter over the 16 lanes of the row group (lane bits 4, 2, 1,
        // 0): at each of the first levels a lane keeps the half of its values
        // selected by its lane bit and adds the partner's copy of that half.
        const int lane = threadIdx.x & 31;
        const int l4 = (lane >> 4) & 1, l2 = (lane >> 2) & 1, l1 = (lane >> 1) & 1;
        float v1[V / 2];
#pragma unroll
        for (int j = 0; j < V / 2; ++j) {
            const float keep = l4 ? v0[V / 2 + j] : v0[j];
            const float send = l4 ? v0[j] : v0[V / 2 + j];
            v1[j] = keep + __shfl_xor_sync(0xffffffffu, send, 16);
        }
        float v2[V / 4];
#pragma unroll
        for (int j = 0; j < V / 4; ++j) {
            const float keep = l2 ? v1[V / 4 + j] : v1[j];
            const float send = l2 ? v1[j] : v1[V / 4 + j];
            v2[j] = keep + __shfl_xor_sync(0xffffffffu, send, 4);
        }
        float v3[A];
        int i_own;
        bool writer;
        if constexpr (NR == 8) {
            // 6 values: one more halving (lane bit 1), then lane bit 0 sums
            // both copies; lanes with bit 0 clear hold row 4 l4 + 2 l2 + l1
#pragma unroll
            for (int j = 0; j < A; ++j) {
                const float keep = l1 ? v2[A + j] : v2[j];
                const float send = l1 ? v2[j] : v2[A + j];
                v3[j] = keep + __shfl_xor_sync(0xffffffffu, send, 2);
            }
#pragma unroll
            for (int j = 0; j < A; ++j) v3[j] += __shfl_xor_sync(0xffffffffu, v3[j], 1);
            i_own = 4 * l4 + 2 * l2 + l1;
            writer = (lane & 1) == 0;
        } else {
            // 3 values (row 2 l4 + l2): lane bits 1 and 0 sum all copies
#pragma unroll
            for (int j = 0; j < A; ++j) v3[j] = v2[j] + __shfl_xor_sync(0xffffffffu, v2[j], 2);
#pragma unroll
            for (int j = 0; j < A; ++j) v3[j] += __shfl_xor_sync(0xffffffffu, v3[j], 1);
            i_own = 2 * l4 + l2;
            writer = (lane & 3) == 0;
        }
        if (writer) {
#pragma unroll
            for (int j = 0; j < A; ++j) LG[(ty + 16 * i_own) * LS + j] = v3[j] + b3[j];
        }
        __syncthreads();
    }
};

// 256-row pass of one policy with H = 64 and 8x8 register tiles (256
// threads): thread (tx, ty), tx = lane % 8 and ty = 4 warp + lane / 8,
// computes rows ty + 32 i (i = 0..7) and columns {4tx..4tx+3} and
// {32+4tx..32+4tx+3}, accumulating column pairs with packed fp32 FMAs. Per k
// a thread issues 2 16-byte weight loads (4 column pairs), 8 duplications of
// an input into a pair and 32 packed FMAs; its 8 inputs arrive as 2 16-byte
// loads amortised over 4 k. A warp's 4 row groups are 4 consecutive rows,
// which the bank-skewed strides (HS = 68, XS = 20 floats) put in different
// banks; its 8 column groups read one 128-byte weight row. Layer 3 is folded
// into layer 2's epilogue: packed dot products over the thread's column pairs,
// then a reduce-scatter over the 8 lanes of a row group after which lane j
// holds the logits of the group's row j.
template <int IN, int A>
struct MlpF32R8 {
    static constexpr int H = 64;
    static constexpr int kThreads = 256;
    static constexpr int kRows = 256;
    static constexpr int XS = (IN + 3) / 4 * 4;
    static constexpr int HS = H + 4;
    static constexpr int LS = (A + 3) / 4 * 4;
    using u64 = unsigned long long;

    __device__ static int col_group() { return threadIdx.x & 7; }
    __device__ static int row_group() { return (threadIdx.x >> 5) * 4 + ((threadIdx.x >> 3) & 3); }

    __device__ static void init(u64 (&acc)[8][4], const float* __restrict__ b, int c0, int c1) {
        const ulonglong2 bA = *reinterpret_cast<const ulonglong2*>(b + c0);
        const ulonglong2 bB = *reinterpret_cast<const ulonglong2*>(b + c1);
#pragma unroll
        for (int i = 0; i < 8; ++i) { acc[i][0] = bA.x; acc[i][1] = bA.y; acc[i][2] = bB.x; acc[i][3] = bB.y; }
    }

    // acc += rows' inputs [4 k from xa] x W rows k0..k0+3 (kk < kmax)
    __device__ static void block(u64 (&acc)[8][4], const float4 (&xa)[8], const float* __restrict__ W,
                                 int k0, int kmax, int c0, int c1) {
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {
            if (kk < kmax) {
                const ulonglong2 wA = *reinterpret_cast<const ulonglong2*>(W + (k0 + kk) * H + c0);
                const ulonglong2 wB = *reinterpret_cast<const ulonglong2*>(W + (k0 + kk) * H + c1);
                u64 x2[8];
#pragma unroll
                for (int i = 0; i < 8; ++i)
                    x2[i] = f2_dup(kk == 0 ? xa[i].x : kk == 1 ? xa[i].y : kk == 2 ? xa[i].z : xa[i].w);
#pragma unroll
                for (int i = 0; i < 8; ++i) f2_fma(acc[i][0], x2[i], wA.x);
#pragma unroll
                for (int i = 0; i < 8; ++i) f2_fma(acc[i][1], x2[i], wA.y);
#pragma unroll
                for (int i = 0; i < 8; ++i) f2_fma(acc[i][2], x2[i], wB.x);
#pragma unroll
                for (int i = 0; i < 8; ++i) f2_fma(acc[i][3], x2[i], wB.y);
            }
        }
    }

    // Layer 1 into H1 (rows of X, XSTRIDE floats apart, 16-byte aligned). Ends
    // with __syncthreads.
    template <int XSTRIDE = XS>
    __device__ static void layer1(const float* __restrict__ X, float* __restrict__ H1,
                                  const float* __restrict__ W1T, const float* __restrict__ b1) {
        const int tx = col_group(), ty = row_group();
        const int c0 = tx * 4, c1 = H / 2 + tx * 4;
        u64 acc[8][4];
        init(acc, b1, c0, c1);
#pragma unroll
        for (int k0 = 0; k0 < IN; k0 += 4) {
            float4 xa[8];
#pragma unroll
            for (int i = 0; i < 8; ++i)
                xa[i] = *reinterpret_cast<const float4*>(X + (ty + 32 * i) * XSTRIDE + k0);
            block(acc, xa, W1T, k0, IN - k0, c0, c1);
        }
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            float* hr = H1 + (ty + 32 * i) * HS;
            const u64 p0 = f2_relu(acc[i][0]), p1 = f2_relu(acc[i][1]);
            const u64 p2 = f2_relu(acc[i][2]), p3 = f2_relu(acc[i][3]);
            *reinterpret_cast<ulonglong2*>(hr + c0) = make_ulonglong2(p0, p1);
            *reinterpret_cast<ulonglong2*>(hr + c1) = make_ulonglong2(p2, p3);
        }
        __syncthreads();
    }

    // Layers 2 and 3: H1 -> logits rows of LG [256][LS]. Ends with __syncthreads.
    __device__ static void layer23(const float* __restrict__ H1, float* __restrict__ LG,
                                   const float* __restrict__ W2T, const float* __restrict__ b2,
                                   const float* __restrict__ W3, const float* __restrict__ b3) {
        const int tx = col_group(), ty = row_group();
        const int c0 = tx * 4, c1 = H / 2 + tx * 4;
        u64 acc[8][4];
        init(acc, b2, c0, c1);
#pragma unroll 4
        for (int k0 = 0; k0 < H; k0 += 4) {
            float4 ha[8];
#pragma unroll
            for (int i = 0; i < 8; ++i)
                ha[i] = *reinterpret_cast<const float4*>(H1 + (ty + 32 * i) * HS + k0);
            block(acc, ha, W2T, k0, 4, c0, c1);
        }
#pragma unroll
        for (int i = 0; i < 8; ++i)
#pragma unroll
            for (int p = 0; p < 4; ++p) acc[i][p] = f2_relu(acc[i][p]);
        constexpr int V = 8 * A;                  // partial logits of this thread
        float v0[V];
#pragma unroll
        for (int a = 0; a < A; ++a) {
            const ulonglong2 wA = *reinterpret_cast<const ulonglong2*>(W3 + a * H + c0);
            const ulonglong2 wB = *reinterpret_cast<const ulonglong2*>(W3 + a * H + c1);
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                u64 t = 0ull;
                f2_fma(t, acc[i][0], wA.x);
                f2_fma(t, acc[i][1], wA.y);
                f2_fma(t, acc[i][2], wB.x);
                f2_fma(t, acc[i][3], wB.y);
                const float2 q = f2_split(t);
                v0[i * A + a] = q.x + q.y;
            }
        }
        // Reduce-scatter over lane bits 2, 1, 0: at each level a lane keeps the
        // half of its values selected by its lane bit and adds the partner's
        // copy of that half; lane j ends with row j's A logits.
        const int lane = threadIdx.x & 31;
        const int l2 = (lane >> 2) & 1, l1 = (lane >> 1) & 1, l0 = lane & 1;
        float v1[V / 2];
#pragma unroll
        for (int j = 0; j < V / 2; ++j) {
            const float keep = l2 ? v0[V / 2 + j] : v0[j];
            const float send = l2 ? v0[j] : v0[V / 2 + j];
            v1[j] = keep + __shfl_xor_sync(0xffffffffu, send, 4);
        }
        float v2[V / 4];
#pragma unroll
        for (int j = 0; j < V / 4; ++j) {
            const float keep = l1 ? v1[V / 4 + j] : v1[j];
            const float send = l1 ? v1[j] : v1[V / 4 + j];
            v2[j] = keep + __shfl_xor_sync(0xffffffffu, send, 2);
        }
        float v3[A];
#pragma unroll
        for (int j = 0; j < A; ++j) {
            const float keep = l0 ? v2[A + j] : v2[j];
            const float send = l0 ? v2[j] : v2[A + j];
            v3[j] = keep + __shfl_xor_sync(0xffffffffu, send, 1);
        }
        float* lr = LG + (ty + 32 * (lane & 7)) * LS;
#pragma unroll
        for (int j = 0; j < A; ++j) lr[j] = v3[j] + b3[j];
        __syncthreads();
    }
};

}  // namespace malib
