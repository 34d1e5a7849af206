// Learner-side update on the device: one independent learner's policy-gradient
// step on the samples a rollout wrote (Sec. 3.3 "Independent Learning": one
// learner per policy, trained on its own agents' experience; App. C.2: the
// training workflow's optimize() with Adam and an entropy coefficient).
//
// For policy p with samples S_p (each (episode, step, environment, agent) whose
// combination gives that agent policy p; M = |S_p|):
//   L = -(1/M) sum_i [ (G_i - b) log pi(a_i | o_i) + beta H(pi(. | o_i)) ],
// G the discounted return-to-go within the episode, b the mean of G over S_p,
// H the entropy of the softmax over the 5 actions. The gradient by the chain
// rule: dL/dz_j = (1/M) [ (G - b)(pi_j - [j = a]) + beta pi_j (log pi_j + H) ],
// back through W3, the ReLUs (pre-activation > 0) and W2, W1.
// The PPO variant (clip > 0; Schulman et al. 2017's clipped surrogate, the
// same advantage A = G - b) replaces (G - b) log pi(a | o) by
// min(rho A, clip(rho, 1 - eps, 1 + eps) A), rho = pi(a | o) / mu(a | o) with mu
// the behavior policy whose logits the rollout recorded; the unclipped term
// carries the gradient A rho (pi_j - [j = a]) where it is the minimum (ties
// to it), the clipped one none.
//
// Kernels, in stream order:
//  1. learn_slots_kernel: the (combination, agent) slots acting with p, in
//     ascending order (one block).
//  2. learn_returns_kernel: G of every sample by the backward recursion
//     G_t = r_t + gamma G_{t+1}, one thread per (slot, episode, env), and
//     per-block fp64 sums of G.
//  3. learn_baseline_kernel: M and b = sum G / M in a fixed order (one block).
//  4. learn_grad_kernel: persistent CTAs over tiles of 128 samples: forward
//     (fp32 FMA, hidden 64), logits, softmax, dL/dz, the backward pass, and
//     the weight gradients accumulated in registers over the CTA's tiles (each
//     thread a 4 x 4 block of dW2 and a few entries of the rest); the tile's
//     activations are stored feature-major in shared memory so that every
//     product reads 16-byte vectors; each CTA writes its partial gradient.
//  5. learn_reduce_kernel: the partials summed over CTAs in a fixed order into
//     the gradient (the malib_policy_desc layout) and the loss statistics.
// Deterministic: no atomics, every sum in a fixed order.
// Adam (Kingma and Ba): learn_adam_kernel, elementwise with bias correction.
#include <cmath>

#include "device_common.cuh"
#include "internal.h"
#include "mlp_f32.cuh"      // packed fp32 pair helpers (f2_fma: two IEEE fmaf per instruction)

namespace malib {

namespace {

constexpr int kH = 64, kA = 5, kTile = 128, kThreads = 256;
// The per-tile activations are stored feature-major ([feature][sample], rows of
// kTS floats, 16-byte aligned), so that a thread's 8 samples or 4 consecutive
// samples are one or two 16-byte loads; kTS = 132 spreads rows 16 apart over
// the banks.
constexpr int kTS = kTile + 4;
constexpr int kXR = kLearnMaxIn;     // observation feature rows

// Shared-memory layout of learn_grad_kernel (floats).
constexpr int kSW1T = 0;                          // [in][64]: W1T[k][j] = W1[j][k]
constexpr int kSB1 = kSW1T + kLearnMaxIn * kH;
constexpr int kSW2T = kSB1 + kH;                  // [64][64]: W2T[k][j] = W2[j][k]
constexpr int kSW2 = kSW2T + kH * kH;             // [64][64]: W2[j][k]
constexpr int kSB2 = kSW2 + kH * kH;
constexpr int kSW3 = kSB2 + kH;                   // [5][64]
constexpr int kSB3 = kSW3 + kA * kH;              // [8]
constexpr int kSX = kSB3 + 8;                     // XT [in][kTS] observations
constexpr int kSH1 = kSX + kXR * kTS;             // H1T [64][kTS] post-ReLU layer 1
constexpr int kSH2 = kSH1 + kH * kTS;             // H2T [64][kTS] post-ReLU layer 2
constexpr int kSD2 = kSH2 + kH * kTS;             // D2T [64][kTS] dL/d(pre-activation 2)
constexpr int kSD1 = kSD2 + kH * kTS;             // D1T [64][kTS] dL/d(pre-activation 1)
constexpr int kSDZ = kSD1 + kH * kTS;             // DZT [8][kTS] dL/dz
constexpr int kSFloats = kSDZ + 8 * kTS;
constexpr size_t kSBytes = (size_t)kSFloats * 4;
static_assert(kSBytes <= 232448, "fits the 227 KB of shared memory of a CTA");
static_assert(kSX % 4 == 0 && kTS % 4 == 0, "16-byte aligned rows");

// One block per policy b of the batch: the slots acting with it, ascending.
__global__ void __launch_bounds__(1024) learn_slots_kernel(LearnArgs a) {
    __shared__ int warp_n[32];
    __shared__ int base;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int b = blockIdx.x;
    const int total = a.n_pairs * a.n_agents;
    const int policy = a.pols[b];
    int32_t* slots = a.slots + (int64_t)b * total;
    if (tid == 0) base = 0;
    __syncthreads();
    for (int c0 = 0; c0 < total; c0 += blockDim.x) {
        const int i = c0 + tid;
        const int pid = i < total ? a.pairs[i] : -1;
        if (b == 0 && i < total && (pid < 0 || pid >= a.n_pol)) atomicOr(a.err, ERRBIT_BAD_PAIR);
        const bool mine = i < total && pid == policy;
        const unsigned m = __ballot_sync(0xffffffffu, mine);
        if (lane == 0) warp_n[warp] = __popc(m);
        __syncthreads();
        int before = base;
        for (int w = 0; w < warp; ++w) before += warp_n[w];
        if (mine) slots[before + __popc(m & ((1u << lane) - 1u))] = i;   // c * n_agents + k
        __syncthreads();
        if (tid == 0) {
            int n = 0;
            for (int w = 0; w < (int)(blockDim.x >> 5); ++w) n += warp_n[w];
            base += n;
        }
        __syncthreads();
    }
    if (tid == 0) a.n_slots[b] = base;
}

// The batch's sample and tile offsets (prefix sums over the policies; one thread).
__global__ void learn_plan_kernel(LearnArgs a) {
    if (threadIdx.x != 0 || blockIdx.x != 0) return;
    const int64_t per_slot = a.n_episodes * a.T * (a.n_envs / a.n_pairs);
    int64_t s = 0, t = 0;
    for (int b = 0; b < a.nb; ++b) {
        a.samp_off[b] = s;
        a.tile_off[b] = t;
        const int64_t M = (int64_t)a.n_slots[b] * per_slot;
        s += M;
        t += (M + 127) / 128;
    }
    a.samp_off[a.nb] = s;
    a.tile_off[a.nb] = t;
}

// Grid (blocks, nb): G of every sample of policy b by the backward recursion
// G_t = r_t + gamma G_{t+1}, one thread per (slot, episode, env), and per-block
// fp64 sums of G.
__global__ void __launch_bounds__(256) learn_returns_kernel(LearnArgs a) {
    __shared__ double red[256];
    const int b = blockIdx.y;
    const int epp = (int)(a.n_envs / a.n_pairs);
    const int64_t n_seq = (int64_t)a.n_slots[b] * a.n_episodes * epp;
    const int32_t* slots = a.slots + (int64_t)b * a.n_pairs * a.n_agents;
    float* G = a.G + a.samp_off[b];
    if ((int64_t)blockIdx.x * blockDim.x >= n_seq) {
        // no sequence of policy b reaches this block: its partial is 0, as the
        // reduction below would give, without the barriers
        if (threadIdx.x == 0) a.gsum[(int64_t)b * gridDim.x + blockIdx.x] = 0.0;
        return;
    }
    double sum = 0.0;
    for (int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; q < n_seq;
         q += (int64_t)gridDim.x * blockDim.x) {
        const int64_t slot = q / (a.n_episodes * epp);
        const int64_t rem = q - slot * a.n_episodes * epp;
        const int64_t e = rem / epp;
        const int r = (int)(rem - e * epp);
        const int ck = slots[slot];
        const int c = ck / a.n_agents, k = ck - c * a.n_agents;
        const int64_t env = (int64_t)c * epp + r;
        // backward over the episode, 8 steps at a time: the 8 rewards are loaded
        // together (the stores to G would otherwise hold each load behind the
        // previous step's store), then the same recurrence in the same order
        float g = 0.f;
        for (int t_hi = a.T; t_hi > 0; t_hi -= 8) {
            float rv[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int t = t_hi - 1 - u;
                rv[u] = t >= 0 ? a.reward[((e * a.T + t) * a.n_envs + env) * a.n_agents + k] : 0.f;
            }
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int t = t_hi - 1 - u;
                if (t >= 0) {
                    g = __fadd_rn(rv[u], __fmul_rn(a.gamma, g));
                    G[((slot * a.n_episodes + e) * a.T + t) * epp + r] = g;
                    sum += (double)g;
                }
            }
        }
    }
    red[threadIdx.x] = sum;
    __syncthreads();
    for (int w = blockDim.x / 2; w > 0; w >>= 1) {
        if ((int)threadIdx.x < w) red[threadIdx.x] += red[threadIdx.x + w];
        __syncthreads();
    }
    if (threadIdx.x == 0) a.gsum[(int64_t)b * gridDim.x + blockIdx.x] = red[0];
}

// One warp per policy b: lane l sums blocks l, l + 32, ... in order, then a
// fixed xor tree; M and the baseline b = sum G / M.
__global__ void learn_baseline_kernel(LearnArgs a, int n_blocks) {
    const int lane = threadIdx.x & 31;
    const int b = blockIdx.x;
    double s = 0.0;
    for (int k = lane; k < n_blocks; k += 32) s += a.gsum[(int64_t)b * n_blocks + k];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    if (threadIdx.x != 0) return;
    const double M = (double)(a.samp_off[b + 1] - a.samp_off[b]);
    a.stats[4 * b] = M;
    a.stats[4 * b + 1] = M > 0 ? s / M : 0.0;
}

// Sample s of the policy's sample order: (slot, episode, step, env) -> the
// trajectory index of its (episode, step, env, agent).
__device__ __forceinline__ int64_t sample_index(const LearnArgs& a, const int32_t* slots, int64_t s, int epp) {
    const int r = (int)(s % epp);
    const int64_t q = s / epp;                        // (slot, e, t)
    const int t = (int)(q % a.T);
    const int64_t q2 = q / a.T;
    const int64_t e = q2 % a.n_episodes, slot = q2 / a.n_episodes;
    const int ck = slots[slot];
    const int c = ck / a.n_agents, ka = ck - c * a.n_agents;
    const int64_t env = (int64_t)c * epp + r;
    return ((e * a.T + t) * a.n_envs + env) * a.n_agents + ka;
}

// H_out[j][s] = relu(b[j] + sum_k W[k][j] H_in[k][s]) for this thread's 8
// samples (8 sg ..) and 4 outputs (ng + 16 q): per k two 16-byte loads of H_in
// (four sample pairs) and four weights, each duplicated into a pair, for 16
// packed FMAs (each lane an fmaf in the same order as a scalar loop).
__device__ __forceinline__ void dense_relu(const float* __restrict__ Win, const float* __restrict__ b,
                                           const float* __restrict__ Hin, int K, float* __restrict__ Hout,
                                           int sg, int ng) {
    using u64 = unsigned long long;
    u64 acc[4][4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const u64 b2 = f2_dup(b[ng + 16 * q]);
#pragma unroll
        for (int i = 0; i < 4; ++i) acc[q][i] = b2;
    }
#pragma unroll 4
    for (int k = 0; k < K; ++k) {
        const ulonglong2 x0 = *reinterpret_cast<const ulonglong2*>(Hin + k * kTS + 8 * sg);
        const ulonglong2 x1 = *reinterpret_cast<const ulonglong2*>(Hin + k * kTS + 8 * sg + 4);
        const u64 x[4] = {x0.x, x0.y, x1.x, x1.y};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const u64 w = f2_dup(Win[k * kH + ng + 16 * q]);
#pragma unroll
            for (int i = 0; i < 4; ++i) f2_fma(acc[q][i], x[i], w);
        }
    }
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        ulonglong2* o = reinterpret_cast<ulonglong2*>(Hout + (ng + 16 * q) * kTS + 8 * sg);
        o[0] = make_ulonglong2(f2_relu(acc[q][0]), f2_relu(acc[q][1]));
        o[1] = make_ulonglong2(f2_relu(acc[q][2]), f2_relu(acc[q][3]));
    }
}

// The 8 values of a sample-pair row (four pairs) where the activations h are
// positive, else 0 (the ReLU's derivative), stored at o.
__device__ __forceinline__ void store_masked(float* __restrict__ o, const unsigned long long (&v)[4],
                                             const float* __restrict__ h) {
    const float4 h0 = *reinterpret_cast<const float4*>(h);
    const float4 h1 = *reinterpret_cast<const float4*>(h + 4);
    const float2 v0 = f2_split(v[0]), v1 = f2_split(v[1]), v2 = f2_split(v[2]), v3 = f2_split(v[3]);
    *reinterpret_cast<float4*>(o) = make_float4(h0.x > 0.f ? v0.x : 0.f, h0.y > 0.f ? v0.y : 0.f,
                                                h0.z > 0.f ? v1.x : 0.f, h0.w > 0.f ? v1.y : 0.f);
    *reinterpret_cast<float4*>(o + 4) = make_float4(h1.x > 0.f ? v2.x : 0.f, h1.y > 0.f ? v2.y : 0.f,
                                                    h1.z > 0.f ? v3.x : 0.f, h1.w > 0.f ? v3.y : 0.f);
}

// A CTA's contiguous share [lo, hi) of the batch's tiles (all policies' tiles
// in policy order).
__device__ __forceinline__ int64_t share_lo(const LearnArgs& a, int64_t c) {
    return a.tile_off[a.nb] * c / a.grid;
}

__global__ void __launch_bounds__(kThreads, 1) learn_grad_kernel(LearnArgs a) {
    extern __shared__ __align__(16) float sm[];
    const int tid = threadIdx.x;
    const int in = a.in;
    const int epp = (int)(a.n_envs / a.n_pairs);
    const int P = kH * in + kH + kH * kH + kH + kA * kH + kA;
    const int64_t lo = share_lo(a, blockIdx.x), hi = share_lo(a, blockIdx.x + 1);

    float* XT = sm + kSX;
    float* H1T = sm + kSH1;
    float* H2T = sm + kSH2;
    float* D2T = sm + kSD2;
    float* D1T = sm + kSD1;
    float* DZT = sm + kSDZ;
    const int sg = tid >> 4, ng = tid & 15;           // layers: samples 8 sg .., outputs ng + 16 q
    // this thread's gradient entries, accumulated over the CTA's tiles
    float gW2[4][4] = {};                              // dW2[ng' + 16 p][kb + 16 q], ng' = sg
    const int w1j = tid & 63, w1k = tid >> 6;          // dW1[w1j][w1k + 4 q]
    float gW1[kLearnMaxIn / 4] = {};
    float gW3[2] = {};                                 // dW3 entries tid, tid + 256 of [5][64]
    float gB = 0.f;                                    // b1 (tid < 64), b2 (64..127), b3 (128..132)
    float lsum = 0.f, hsum = 0.f;                      // loss and entropy of this thread's samples
    int b = -1;                                        // the batch's policy of the current tiles
    int64_t M = 0, t0 = 0;
    float invM = 0.f, base = 0.f;
    const int32_t* slots = nullptr;
    const float* Gb = nullptr;
    // this CTA's partial gradient of policy b, in the malib_policy_desc layout:
    // W1 [64][in], b1, W2 [64][64], b2, W3 [5][64], b3, then loss and entropy sums
    auto flush = [&]() {
        float* out = a.gpart + ((int64_t)b * a.grid + blockIdx.x) * (P + 2);
#pragma unroll
        for (int q = 0; q < kLearnMaxIn / 4; ++q) {
            const int k = w1k + 4 * q;
            if (k < in) out[w1j * in + k] = gW1[q];
        }
        const int oW2 = kH * in + kH;
#pragma unroll
        for (int p = 0; p < 4; ++p)
#pragma unroll
            for (int q = 0; q < 4; ++q) out[oW2 + (sg + 16 * p) * kH + ng + 16 * q] = gW2[p][q];
        const int oW3 = oW2 + kH * kH + kH;
#pragma unroll
        for (int q = 0; q < 2; ++q) {
            const int e = tid + kThreads * q;
            if (e < kA * kH) out[oW3 + e] = gW3[q];
        }
        if (tid < kH) out[kH * in + tid] = gB;                          // b1
        else if (tid < 2 * kH) out[oW2 + kH * kH + tid - kH] = gB;      // b2
        else if (tid < 2 * kH + kA) out[oW3 + kA * kH + tid - 2 * kH] = gB;   // b3
        // loss and entropy sums (fixed-order tree in shared memory; the tiles'
        // buffers are free between tiles)
        float* red = sm + kSX;
        red[tid] = lsum;
        red[kThreads + tid] = hsum;
        __syncthreads();
        for (int w = kThreads / 2; w > 0; w >>= 1) {
            if (tid < w) {
                red[tid] += red[tid + w];
                red[kThreads + tid] += red[kThreads + tid + w];
            }
            __syncthreads();
        }
        if (tid == 0) {
            out[P] = red[0];
            out[P + 1] = red[kThreads];
        }
        __syncthreads();
    };
    for (int64_t tile = lo; tile < hi; ++tile) {
        if (b < 0 || tile >= a.tile_off[b + 1]) {
            // the next policy of the batch with tiles: flush the previous one's
            // partials, stage this one (F32Layout: W1T [in][64], b1, W2T [64][64],
            // b2, W3 [5][64], b3), restart the sums
            if (b >= 0) flush();
            if (b < 0) b = 0;
            while (tile >= a.tile_off[b + 1]) ++b;
            const float* pol = a.arena + a.pol_offs[b];
            for (int i = tid; i < in * kH; i += kThreads) sm[kSW1T + i] = pol[i];
            for (int i = tid; i < kH; i += kThreads) sm[kSB1 + i] = pol[in * kH + i];
            for (int i = tid; i < kH * kH; i += kThreads) {
                const float w = pol[in * kH + kH + i];               // W2T[k][j], i = k * 64 + j
                sm[kSW2T + i] = w;
                sm[kSW2 + (i & (kH - 1)) * kH + (i >> 6)] = w;        // W2[j][k]
            }
            for (int i = tid; i < kH; i += kThreads) sm[kSB2 + i] = pol[in * kH + kH + kH * kH + i];
            for (int i = tid; i < kA * kH; i += kThreads) sm[kSW3 + i] = pol[in * kH + 2 * kH + kH * kH + i];
            if (tid < kA) sm[kSB3 + tid] = pol[in * kH + 2 * kH + kH * kH + kA * kH + tid];
            M = a.samp_off[b + 1] - a.samp_off[b];
            invM = M > 0 ? (float)(1.0 / (double)M) : 0.f;
            base = (float)a.stats[4 * b + 1];
            slots = a.slots + (int64_t)b * a.n_pairs * a.n_agents;
            Gb = a.G + a.samp_off[b];
            t0 = a.tile_off[b];
#pragma unroll
            for (int p = 0; p < 4; ++p)
#pragma unroll
                for (int q = 0; q < 4; ++q) gW2[p][q] = 0.f;
#pragma unroll
            for (int q = 0; q < kLearnMaxIn / 4; ++q) gW1[q] = 0.f;
            gW3[0] = gW3[1] = 0.f;
            gB = 0.f;
            lsum = hsum = 0.f;
            __syncthreads();
        }
        const int64_t s0 = (tile - t0) * kTile;
        // the tile's observations (feature-major; zero columns past M), and for
        // the logits phase each sample's action and return
        int act = 0;
        float ret = 0.f, lmu = 0.f;
        {
            const int r = tid & (kTile - 1), half = tid >> 7;
            const int64_t s = s0 + r;
            if (s < M) {
                const int64_t ix = sample_index(a, slots, s, epp);
                const float* orow = a.obs + ix * a.xs;
                for (int k = half; k < in; k += 2) XT[k * kTS + r] = orow[k];
                if (half == 0) {
                    act = a.action[ix];
                    ret = Gb[s];
                    if (a.clip > 0.f) {
                        // log mu(a | o): the behavior policy's log-softmax at the action taken
                        const float* bl = a.blogits + ix * kA;
                        float l[kA];
#pragma unroll
                        for (int j = 0; j < kA; ++j) l[j] = bl[j];
                        float m = l[0];
#pragma unroll
                        for (int j = 1; j < kA; ++j) m = fmaxf(m, l[j]);
                        float S = 0.f;
#pragma unroll
                        for (int j = 0; j < kA; ++j) S += expf(l[j] - m);
                        float la = l[0];
#pragma unroll
                        for (int j = 1; j < kA; ++j)
                            if (j == act) la = l[j];
                        lmu = la - m - logf(S);
                    }
                }
            } else {
                for (int k = half; k < in; k += 2) XT[k * kTS + r] = 0.f;
            }
        }
        __syncthreads();
        dense_relu(sm + kSW1T, sm + kSB1, XT, in, H1T, sg, ng);
        __syncthreads();
        dense_relu(sm + kSW2T, sm + kSB2, H1T, kH, H2T, sg, ng);
        __syncthreads();
        // logits, softmax and dL/dz, one sample per thread (threads 0 .. 127)
        if (tid < kTile) {
            const int64_t s = s0 + tid;
            float dz[kA] = {0.f, 0.f, 0.f, 0.f, 0.f};
            if (s < M) {
                const float adv = ret - base;
                float z[kA];
#pragma unroll
                for (int j = 0; j < kA; ++j) z[j] = sm[kSB3 + j];
#pragma unroll 8
                for (int h = 0; h < kH; ++h) {
                    const float x = H2T[h * kTS + tid];
#pragma unroll
                    for (int j = 0; j < kA; ++j) z[j] = fmaf(sm[kSW3 + j * kH + h], x, z[j]);
                }
                float m = z[0];
#pragma unroll
                for (int j = 1; j < kA; ++j) m = fmaxf(m, z[j]);
                float S = 0.f;
#pragma unroll
                for (int j = 0; j < kA; ++j) S += expf(z[j] - m);
                const float lS = logf(S);
                float logp[kA], pi[kA], H = 0.f;
#pragma unroll
                for (int j = 0; j < kA; ++j) {
                    logp[j] = z[j] - m - lS;
                    pi[j] = expf(logp[j]);
                    H -= pi[j] * logp[j];
                }
                float lp_a = logp[0];
#pragma unroll
                for (int j = 1; j < kA; ++j)
                    if (j == act) lp_a = logp[j];
                if (a.clip > 0.f) {
                    // PPO: min(rho A, clip(rho) A); the unclipped term carries the
                    // gradient A rho (pi - [j = a]) when it is the minimum (ties to it)
                    const float rho = expf(lp_a - lmu);
                    const float unc = rho * adv;
                    const float clp = fminf(fmaxf(rho, 1.f - a.clip), 1.f + a.clip) * adv;
                    const float w = unc <= clp ? unc : 0.f;
#pragma unroll
                    for (int j = 0; j < kA; ++j)
                        dz[j] = (w * (pi[j] - (j == act ? 1.f : 0.f)) + a.beta * pi[j] * (logp[j] + H)) * invM;
                    lsum -= fminf(unc, clp) + a.beta * H;
                } else {
#pragma unroll
                    for (int j = 0; j < kA; ++j)
                        dz[j] = (adv * (pi[j] - (j == act ? 1.f : 0.f)) + a.beta * pi[j] * (logp[j] + H)) * invM;
                    lsum -= adv * lp_a + a.beta * H;
                }
                hsum += H;
            }
#pragma unroll
            for (int j = 0; j < kA; ++j) DZT[j * kTS + tid] = dz[j];
        }
        __syncthreads();
        // D2 = (dz W3) * [h2 > 0]: samples 8 sg .. (four pairs), units ng + 16 q
        {
            using u64 = unsigned long long;
            u64 dzv[kA][4];
#pragma unroll
            for (int c = 0; c < kA; ++c) {
                const ulonglong2 d0 = *reinterpret_cast<const ulonglong2*>(DZT + c * kTS + 8 * sg);
                const ulonglong2 d1 = *reinterpret_cast<const ulonglong2*>(DZT + c * kTS + 8 * sg + 4);
                dzv[c][0] = d0.x; dzv[c][1] = d0.y; dzv[c][2] = d1.x; dzv[c][3] = d1.y;
            }
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int j = ng + 16 * q;
                u64 v[4] = {0ull, 0ull, 0ull, 0ull};
#pragma unroll
                for (int c = 0; c < kA; ++c) {
                    const u64 w = f2_dup(sm[kSW3 + c * kH + j]);
#pragma unroll
                    for (int i = 0; i < 4; ++i) f2_fma(v[i], dzv[c][i], w);
                }
                store_masked(D2T + j * kTS + 8 * sg, v, H2T + j * kTS + 8 * sg);
            }
        }
        __syncthreads();
        // D1 = (D2 W2) * [h1 > 0]: samples 8 sg .. (four pairs), units ng + 16 q
        {
            using u64 = unsigned long long;
            u64 acc[4][4] = {};
#pragma unroll 4
            for (int j = 0; j < kH; ++j) {
                const ulonglong2 d0 = *reinterpret_cast<const ulonglong2*>(D2T + j * kTS + 8 * sg);
                const ulonglong2 d1 = *reinterpret_cast<const ulonglong2*>(D2T + j * kTS + 8 * sg + 4);
                const u64 d[4] = {d0.x, d0.y, d1.x, d1.y};
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const u64 w = f2_dup(sm[kSW2 + j * kH + ng + 16 * q]);
#pragma unroll
                    for (int i = 0; i < 4; ++i) f2_fma(acc[q][i], d[i], w);
                }
            }
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int k = ng + 16 * q;
                store_masked(D1T + k * kTS + 8 * sg, acc[q], H1T + k * kTS + 8 * sg);
            }
        }
        __syncthreads();
        // the tile's weight gradients, 4 samples per 16-byte load; packed pairs
        // of consecutive samples (the even and odd samples' sums, added at the
        // tile's end)
        {
            using u64 = unsigned long long;
            u64 t2[4][4] = {};
#pragma unroll 2
            for (int s = 0; s < kTile; s += 4) {
                ulonglong2 d[4], h[4];
#pragma unroll
                for (int p = 0; p < 4; ++p) {
                    d[p] = *reinterpret_cast<const ulonglong2*>(D2T + (sg + 16 * p) * kTS + s);
                    h[p] = *reinterpret_cast<const ulonglong2*>(H1T + (ng + 16 * p) * kTS + s);
                }
#pragma unroll
                for (int p = 0; p < 4; ++p)
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        f2_fma(t2[p][q], d[p].x, h[q].x);
                        f2_fma(t2[p][q], d[p].y, h[q].y);
                    }
            }
#pragma unroll
            for (int p = 0; p < 4; ++p)
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const float2 v = f2_split(t2[p][q]);
                    gW2[p][q] += v.x + v.y;
                }
        }
        {
            using u64 = unsigned long long;
            u64 t1[kLearnMaxIn / 4] = {};
            for (int s = 0; s < kTile; s += 4) {
                const ulonglong2 d = *reinterpret_cast<const ulonglong2*>(D1T + w1j * kTS + s);
#pragma unroll
                for (int q = 0; q < kLearnMaxIn / 4; ++q) {
                    const int k = w1k + 4 * q;
                    if (k < in) {
                        const ulonglong2 x = *reinterpret_cast<const ulonglong2*>(XT + k * kTS + s);
                        f2_fma(t1[q], d.x, x.x);
                        f2_fma(t1[q], d.y, x.y);
                    }
                }
            }
#pragma unroll
            for (int q = 0; q < kLearnMaxIn / 4; ++q) {
                const float2 v = f2_split(t1[q]);
                gW1[q] += v.x + v.y;
            }
        }
#pragma unroll
        for (int q = 0; q < 2; ++q) {
            const int e = tid + kThreads * q;
            if (e < kA * kH) {
                const int c = e / kH, j = e - c * kH;
                unsigned long long t3 = 0ull;
                for (int s = 0; s < kTile; s += 4) {
                    const ulonglong2 d = *reinterpret_cast<const ulonglong2*>(DZT + c * kTS + s);
                    const ulonglong2 x = *reinterpret_cast<const ulonglong2*>(H2T + j * kTS + s);
                    f2_fma(t3, d.x, x.x);
                    f2_fma(t3, d.y, x.y);
                }
                const float2 v = f2_split(t3);
                gW3[q] += v.x + v.y;
            }
        }
        if (tid < 2 * kH + kA) {
            const float* row = tid < kH ? D1T + tid * kTS : tid < 2 * kH ? D2T + (tid - kH) * kTS
                                                                         : DZT + (tid - 2 * kH) * kTS;
            float g = gB;
            for (int s = 0; s < kTile; s += 4) {
                const float4 d = *reinterpret_cast<const float4*>(row + s);
                g += d.x;
                g += d.y;
                g += d.z;
                g += d.w;
            }
            gB = g;
        }
        __syncthreads();                        // the tile's buffers are rewritten next
    }

    if (b >= 0) flush();
}

// Grid (blocks, nb): policy b's gradient as the sum, in CTA order, of the
// partials of the CTAs whose tile share meets b's tiles (eight interleaved
// partial sums, combined in a fixed order); its loss and mean entropy.
__global__ void learn_reduce_kernel(LearnArgs a, int P) {
    const int j = blockIdx.x * blockDim.x + threadIdx.x;
    const int b = blockIdx.y;
    if (j >= P + 2) return;
    const int64_t t_lo = a.tile_off[b], t_hi = a.tile_off[b + 1];
    int c_lo = 0, c_hi = 0;                  // CTAs [c_lo, c_hi) hold partials of b
    if (t_hi > t_lo) {
        // c_lo: the first CTA whose share ends past t_lo; c_hi: the first CTA
        // after it whose share starts at or past t_hi (or the grid's end). Both
        // start from the shares' proportional position and step to the exact one.
        const int64_t n_t = a.tile_off[a.nb];
        c_lo = (int)min((int64_t)a.grid - 1, t_lo * a.grid / n_t);
        while (c_lo > 0 && share_lo(a, c_lo) > t_lo) --c_lo;
        while (share_lo(a, c_lo + 1) <= t_lo) ++c_lo;
        c_hi = (int)max((int64_t)c_lo + 1, min((int64_t)a.grid, (t_hi * a.grid + n_t - 1) / n_t));
        while (c_hi > c_lo + 1 && share_lo(a, c_hi - 1) >= t_hi) --c_hi;
        while (c_hi < a.grid && share_lo(a, c_hi) < t_hi) ++c_hi;
    }
    // (a CTA with an empty share wrote no partial: it is skipped)
    const float* part = a.gpart + (int64_t)b * a.grid * (P + 2) + j;
    double p8[8] = {0.0, 0.0, 0.0, 0.0, 0.0, 0.0, 0.0, 0.0};
    int u = 0;
    int64_t s_c = share_lo(a, c_lo);
    for (int c = c_lo; c < c_hi; ++c) {
        const int64_t s_n = share_lo(a, c + 1);
        if (s_n > s_c) {
            p8[u] += (double)part[(int64_t)c * (P + 2)];
            u = (u + 1) & 7;
        }
        s_c = s_n;
    }
    const double s = ((p8[0] + p8[1]) + (p8[2] + p8[3])) + ((p8[4] + p8[5]) + (p8[6] + p8[7]));
    double* st = a.stats + 4 * b;
    if (j < P) a.grad[(int64_t)b * P + j] = (float)s;
    else if (j == P) st[2] = st[0] > 0 ? s / st[0] : 0.0;   // loss: (1/M) sum of -(A log pi + beta H)
    else st[3] = st[0] > 0 ? s / st[0] : 0.0;              // mean entropy
}

__global__ void learn_adam_kernel(float* p, const float* g, float* m, float* v, int64_t n, float lr, float b1,
                                  float b2, float eps, float c1, float c2) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        const float gi = g[i];
        const float mi = b1 * m[i] + (1.f - b1) * gi;
        const float vi = b2 * v[i] + (1.f - b2) * gi * gi;
        m[i] = mi;
        v[i] = vi;
        p[i] -= lr * (mi / c1) / (sqrtf(vi / c2) + eps);
    }
}

}  // namespace

int64_t learn_param_count(int in) { return (int64_t)kH * in + kH + kH * kH + kH + kA * kH + kA; }

bool learn_supported(int in, int h1, int h2, int n_actions) {
    return in >= 1 && in <= kLearnMaxIn && h1 == kH && h2 == kH && n_actions == kA;
}

// Upper bounds of the work space (bytes, each region on a 256-byte boundary):
// the distinct policies of a batch own disjoint slots, so their samples together
// are at most every (episode, step, env, agent).
int64_t learn_work_bytes(int32_t nb, int32_t n_pairs, int32_t n_agents, int64_t n_envs, int64_t n_episodes,
                         int32_t T, int in, int grid, int ret_blocks) {
    auto up = [](int64_t b) { return (b + 255) / 256 * 256; };
    const int64_t slots = (int64_t)n_pairs * n_agents;
    const int64_t samples = slots * n_episodes * T * (n_envs / n_pairs);
    return up((int64_t)nb * 4) + up((int64_t)nb * 8) + up((int64_t)nb * slots * 4) + up((int64_t)nb * 4) +
           2 * up((int64_t)(nb + 1) * 8) + up(samples * 4) + up((int64_t)nb * ret_blocks * 8) +
           up((int64_t)nb * 4 * 8) + up((int64_t)nb * grid * (learn_param_count(in) + 2) * 4);
}

void learn_work_layout(uint8_t* base, int32_t nb, int32_t n_pairs, int32_t n_agents, int64_t n_envs,
                       int64_t n_episodes, int32_t T, int in, int grid, int ret_blocks, LearnArgs* a) {
    int64_t off = 0;
    auto take = [&](int64_t bytes) {
        uint8_t* p = base + off;
        off += (bytes + 255) / 256 * 256;
        return p;
    };
    const int64_t slots = (int64_t)n_pairs * n_agents;
    const int64_t samples = slots * n_episodes * T * (n_envs / n_pairs);
    a->pols = reinterpret_cast<int32_t*>(take((int64_t)nb * 4));
    a->pol_offs = reinterpret_cast<int64_t*>(take((int64_t)nb * 8));
    a->slots = reinterpret_cast<int32_t*>(take((int64_t)nb * slots * 4));
    a->n_slots = reinterpret_cast<int32_t*>(take((int64_t)nb * 4));
    a->samp_off = reinterpret_cast<int64_t*>(take((int64_t)(nb + 1) * 8));
    a->tile_off = reinterpret_cast<int64_t*>(take((int64_t)(nb + 1) * 8));
    a->G = reinterpret_cast<float*>(take(samples * 4));
    a->gsum = reinterpret_cast<double*>(take((int64_t)nb * ret_blocks * 8));
    a->stats = reinterpret_cast<double*>(take((int64_t)nb * 4 * 8));
    a->gpart = reinterpret_cast<float*>(take((int64_t)nb * grid * (learn_param_count(in) + 2) * 4));
    a->nb = nb;
    a->grid = grid;
}

cudaError_t launch_learn_pg(const LearnArgs& a, int ret_blocks, cudaStream_t s, cudaEvent_t g0, cudaEvent_t g1) {
    if (a.nb <= 0) return cudaSuccess;
    learn_slots_kernel<<<a.nb, 1024, 0, s>>>(a);
    learn_plan_kernel<<<1, 32, 0, s>>>(a);
    learn_returns_kernel<<<dim3(ret_blocks, a.nb), 256, 0, s>>>(a);
    learn_baseline_kernel<<<a.nb, 32, 0, s>>>(a, ret_blocks);
    cudaError_t err = cudaFuncSetAttribute(learn_grad_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           (int)kSBytes);
    if (err != cudaSuccess) return err;
    if (g0) cudaEventRecord(g0, s);
    learn_grad_kernel<<<a.grid, kThreads, kSBytes, s>>>(a);
    if (g1) cudaEventRecord(g1, s);
    const int P = (int)learn_param_count(a.in);
    learn_reduce_kernel<<<dim3((P + 2 + 255) / 256, a.nb), 256, 0, s>>>(a, P);
    return cudaGetLastError();
}

cudaError_t launch_learn_adam(float* p, const float* g, float* m, float* v, int64_t n, float lr, float b1,
                              float b2, float eps, float c1, float c2, int n_sm, cudaStream_t s) {
    if (n == 0) return cudaSuccess;
    int64_t blocks = (n + 255) / 256;
    if (blocks > 4 * (int64_t)n_sm) blocks = 4 * (int64_t)n_sm;
    learn_adam_kernel<<<(unsigned)blocks, 256, 0, s>>>(p, g, m, v, n, lr, b1, b2, eps, c1, c2);
    return cudaGetLastError();
}

}  // namespace malib
