// Batched rollout of cooperative particle spread with bf16 MLP policies on the
// tensor cores (Sec. 3.1 rollout under a policy combination; App. B.1 simple
// spread), for N = 8 agents with 34-float observations and 34-256-256-5 MLPs.
//
// One CTA serves a combination (one block of up to 128 environments) alone.
// Its engine runs all 8 agents' 128-row tiles, restaging the acting agent's
// policy image (bf16 weights and biases, ~162 KB) between agents; the
// population stays resident in L2. A step takes the agents in the order 0..7
// on even steps and 7..0 on odd ones, so it starts with the policy the
// previous step ended with (7 restages per step; none when two agents share a
// policy). Each CTA has 16 warps in three roles:
//  * warps 0-7, the engine: for each agent, the tiles of both episodes
//    through the tensor-core MLP (hidden activations in tensor memory); each
//    row's 5 logits go to shared memory, announced on a per-buffer mbarrier.
//    Layer 2 is issued by the tile's group's first thread, which waits for
//    those logits anyway;
//  * warps 8-11 and 12-15, environment groups 0 and 1: two episodes of the
//    combination in flight, one environment per thread, state in registers.
//    For each agent a group builds its observations (a bf16 tile in one of two
//    buffers, so it stays one agent ahead of the engine; each thread stores
//    its fp32 row, one 144-byte run, to the trajectory), draws the agent's
//    actions from the engine's logits with the (episode, step, agent) Philox
//    keys, and once all 8 agents have acted steps its environments and writes
//    the rewards and done flags.
// An earlier design (8-CTA clusters, CTA k holding agent k's policy, actions
// exchanged by asynchronous stores into peers' shared memory) fitted only 15
// clusters (120 SMs) and replicated every transition 8 times. Every wait is
// bounded.
#include "device_common.cuh"
#include "internal.h"
#include "mlp_tc.cuh"
#include "spread_env.cuh"

namespace malib {

namespace {

constexpr int kN = 8;                        // agents = landmarks
constexpr int kObs = 34, kObsPad = 36, kK1 = 48, kA = 5;
using Eng = MlpTc<kK1, 256, 16, true, /*kBarId=*/1>;    // biases staged with the weights
constexpr int kThreads = 512;
constexpr int kEngineThreads = 256;
// registers per thread after setmaxnreg: the engine's two warpgroups and the two
// environment groups' (whose 8-agent steps and observations need more), summing
// to the launch's 128 per thread
constexpr int kRegLaunch = 128, kRegEngine = 120, kRegEnv = 136;
static_assert(kRegEngine + kRegEnv == 2 * kRegLaunch, "register split within the launch's allocation");

constexpr int kGroups = 2;
constexpr int kLgStride = kA;                                     // logits row stride (floats)
constexpr uint32_t kX = Eng::kSmemBytes;                          // X tiles [group][buffer]
constexpr uint32_t kLgs = kX + kGroups * 2 * Eng::kXBytes;        // logits [group][buffer][env][5]
constexpr uint32_t kActS = kLgs + kGroups * 2 * 128 * kLgStride * 4;   // actions [group][agent][env]
constexpr uint32_t kSmem = kActS + kGroups * kN * 128;
static_assert(kX % 16 == 0 && kLgs % 16 == 0 && kActS % 16 == 0, "16-byte aligned regions");
static_assert(kSmem <= 227 * 1024, "fits one CTA's shared memory");

__device__ __forceinline__ void group_sync(int g) {
    if (g == 0) asm volatile("bar.sync 2, 128;" ::: "memory");
    else asm volatile("bar.sync 3, 128;" ::: "memory");
}

// A CTA's items, (combination, episode) pairs in order, are taken two at a
// time: group 0 the first, group 1 the next one when it belongs to the same
// combination (else group 1 idles that round). Every role walks the same rounds.
struct Round {
    int pair;
    int64_t ep[kGroups];        // -1: the group idles
    int64_t next;
};

__device__ __forceinline__ Round round_at(int64_t it, int64_t hi, int64_t n_ep) {
    Round r;
    r.pair = (int)(it / n_ep);
    r.ep[0] = it - (int64_t)r.pair * n_ep;
    const bool b = it + 1 < hi && (it + 1) / n_ep == r.pair;
    r.ep[1] = b ? r.ep[0] + 1 : -1;
    r.next = it + (b ? 2 : 1);
    return r;
}

__device__ __forceinline__ bool pair_valid(const RolloutArgs& a, int pair) {
    bool ok = true;                  // every role checks all 8 ids: same decision
    for (int i = 0; i < kN; ++i) {
        const int p = a.pairs[pair * kN + i];
        ok = ok && p >= 0 && p < a.n_pol;
    }
    return ok;
}

// kContact: the agents also push each other apart (soft contact forces).
// kLogits: the call records the logits (the recording code is compiled out of
// the other instances).
template <bool kContact, bool kLogits>
__global__ void __launch_bounds__(kThreads, 1) spread_rollout_tc_kernel(RolloutArgs a) {
    extern __shared__ __align__(128) uint8_t smem[];
    __shared__ __align__(8) uint64_t stage_bar;             // W1 and the biases staged
    __shared__ __align__(8) uint64_t w2_bar;                // W2 and W3 staged
    __shared__ __align__(8) uint64_t mma_bar[2];
    __shared__ __align__(8) uint64_t x_full[kGroups][2];    // a group's tile in buffer b is ready
    __shared__ __align__(8) uint64_t lg_full[kGroups][2];   // the logits of that tile are ready
    __shared__ __align__(8) uint64_t h1_bar[kGroups][2];    // h1 halves of a group's tile stored
    __shared__ uint32_t tmem_base;

    float* lgs = reinterpret_cast<float*>(smem + kLgs);
    uint8_t* acts = smem + kActS;
    const int tid = threadIdx.x, warp = tid >> 5;

    if (tid == 0) {
        mbar_init(&stage_bar, 1);
        mbar_init(&w2_bar, 1);
        mbar_init(&mma_bar[0], 1);
        mbar_init(&mma_bar[1], 1);
        for (int g = 0; g < kGroups; ++g) {
            mbar_init(&h1_bar[g][0], 1);
            mbar_init(&h1_bar[g][1], 1);
            for (int b = 0; b < 2; ++b) {
                mbar_init(&x_full[g][b], 1);
                mbar_init(&lg_full[g][b], 1);
            }
        }
    }
    if (warp == 0) {
        tc::tmem_alloc(&tmem_base, Eng::kTmemCols);
        tc::tmem_relinquish();
    }
    for (uint32_t i = tid * 16; i < kGroups * 2 * Eng::kXBytes; i += kThreads * 16)
        *reinterpret_cast<uint4*>(smem + kX + i) = make_uint4(0, 0, 0, 0);
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    const uint32_t tbase = tmem_base;

    const int epp = (int)(a.n_envs / a.n_pairs);
    const int T = a.episode_len;
    const int64_t items = (int64_t)a.n_pairs * a.n_episodes;
    const int64_t per = (items + gridDim.x - 1) / gridDim.x;
    const int64_t lo = (int64_t)blockIdx.x * per, hi = min(items, lo + per);

    if (warp < 8) {
        // ------------------------------------------------------------ engine
        tc::set_max_regs<kRegEngine, kRegLaunch>();
        uint32_t stage_par = 0, mma_par = 0, x_bits = 0;   // x_full[g][b] phase: bit 2 g + b
        int staged = -1;                                   // policy id in shared memory
        for (int64_t it = lo; it < hi;) {
            const Round rd = round_at(it, hi, a.n_episodes);
            it = rd.next;
            if (!pair_valid(a, rd.pair)) {
                if (tid == 0) atomicOr(a.err, ERRBIT_BAD_PAIR);
                continue;
            }
            for (int t = 0; t < T; ++t) {
                for (int idx = 0; idx < kN; ++idx) {
                    const int k = (t & 1) ? kN - 1 - idx : idx;
                    const int pol = a.pairs[rd.pair * kN + k];
                    if (pol != staged) {
                        // the forwards of the previous agent are complete (each ends
                        // with an engine barrier): restage, W1 and the biases on
                        // stage_bar, which every engine thread waits for, W2 and W3
                        // on w2_bar, which only the MMA thread waits for, before
                        // layer 2 of the next forward
                        if (tid == 0) {
                            fence_proxy_async_smem();
                            const uint8_t* src = reinterpret_cast<const uint8_t*>(a.arena + a.pol_offset[pol]);
                            mbar_arrive_expect_tx(&stage_bar, Eng::kW2 + (Eng::kStageBytes - Eng::kBias));
                            bulk_g2s(smem, src, Eng::kW2, &stage_bar);
                            bulk_g2s(smem + Eng::kBias, src + Eng::kBias, Eng::kStageBytes - Eng::kBias, &stage_bar);
                            mbar_arrive_expect_tx(&w2_bar, Eng::kBias - Eng::kW2);
                            for (uint32_t off = Eng::kW2; off < Eng::kBias; off += 32768u)
                                bulk_g2s(smem + off, src + off, min(32768u, Eng::kBias - off), &w2_bar);
                        }
                        if (!mbar_wait_bounded(&stage_bar, stage_par, kWaitLimitNs) && tid == 0)
                            atomicOr(a.err, ERRBIT_TIMEOUT);
                        stage_par ^= 1u;
                        staged = pol;
                        tc::fence_before_sync();
                        Eng::sync();
                    }
                    const int b = idx & 1;
                    for (int g = 0; g < kGroups; ++g) {
                        if (rd.ep[g] < 0) continue;
                        const uint32_t bit = 1u << (2 * g + b);
                        if (tid == 0 && !mbar_wait_bounded(&x_full[g][b], (x_bits & bit) ? 1u : 0u,
                                                           kWaitLimitNs))
                            atomicOr(a.err, ERRBIT_TIMEOUT);
                        x_bits ^= bit;
                        Eng::sync();
                        float* lgg = lgs + (g * 2 + b) * 128 * kLgStride;
                        Eng::forward(smem, nullptr, tbase, mma_bar, mma_par, a.err,
                                     [&](int row, const float* lg) {
#pragma unroll
                                         for (int j = 0; j < kA; ++j) lgg[row * kLgStride + j] = lg[j];
                                     },
                                     smem_u32(smem + kX + (g * 2 + b) * Eng::kXBytes), /*x_published=*/true,
                                     h1_bar[g], &w2_bar, stage_par ^ 1u, /*helper_all=*/true);
                        // the forward ends with an engine barrier: every row's logits are stored
                        if (tid == 0) mbar_arrive_release(&lg_full[g][b]);
                    }
                }
            }
        }
    } else {
        tc::set_max_regs<kRegEnv, kRegLaunch>();
        // ------------------------------------------------------------ environment groups
        const int g = (warp - 8) >> 2;
        const int e = tid - kEngineThreads - g * 128;     // environment within the block
        uint32_t lg_bits = 0;                              // lg_full[g][b] phase: bit b
        uint32_t h1_par = 0, h1_part = 0;
        uint8_t* ag = acts + g * kN * 128;
        for (int64_t it = lo; it < hi;) {
            const Round rd = round_at(it, hi, a.n_episodes);
            it = rd.next;
            if (!pair_valid(a, rd.pair) || rd.ep[g] < 0) continue;
            const int64_t ep = rd.ep[g];
            const bool mine = e < epp;
            const int64_t env = (int64_t)rd.pair * epp + e;
            const uint64_t gid = (uint64_t)ep * (uint64_t)a.n_envs + (uint64_t)env;
            SpreadEnv<kN> s;
            if (mine) spread_reset<kN>(s, gid, a.seed);
            for (int t = 0; t < T; ++t) {
                const int64_t ix = ((ep * T + t) * a.n_envs + env) * kN;
                // draws the actions of the agent at position j of this step's order
                auto consume = [&](int j) {
                    const int kj = (t & 1) ? kN - 1 - j : j;
                    const int bj = j & 1;
                    const uint32_t par = (lg_bits >> bj) & 1u;
                    if (e == 0) {
                        // while it waits, the group's first thread issues layer 2 of
                        // the group's tile, in two parts as the engine stores h1's
                        // halves in tensor memory (the engine's MMA thread is then
                        // free for its epilogue share); the forward needs it to finish
                        const uint64_t t0 = globaltimer_ns();
                        bool done = false;
                        while (!done) {
                            if (mbar_try_wait(&h1_bar[g][h1_part], (h1_par >> h1_part) & 1u)) {
                                h1_par ^= 1u << h1_part;
                                tc::fence_after_sync();
                                Eng::issue_layer2(smem, tbase, &mma_bar[0], (int)h1_part);
                                h1_part ^= 1u;
                            }
                            done = mbar_try_wait(&lg_full[g][bj], par);
                            if (!done && globaltimer_ns() - t0 > kWaitLimitNs) {
                                atomicOr(a.err, ERRBIT_TIMEOUT);
                                break;
                            }
                        }
                    } else {
                        // an expired wait is recorded by the group's first thread
                        (void)mbar_wait_bounded(&lg_full[g][bj], par, kWaitLimitNs);
                    }
                    lg_bits ^= 1u << bj;
                    if (mine) {
                        const float* lp = lgs + ((g * 2 + bj) * 128 + e) * kLgStride;
                        float l5[kA];
#pragma unroll
                        for (int q = 0; q < kA; ++q) l5[q] = lp[q];
                        const float u = u24(draw(gid, (uint32_t)t, (uint32_t)kj, a.seed).x);
                        const int act = sample_masked<kA>(l5, 0x1Fu, u);
                        if (kLogits)
#pragma unroll
                            for (int q = 0; q < kA; ++q) a.logits[(ix + kj) * kA + q] = l5[q];
                        a.action[ix + kj] = (uint8_t)act;
                        ag[kj * 128 + e] = (uint8_t)act;
                    }
                };
                for (int idx = 0; idx < kN; ++idx) {
                    const int k = (t & 1) ? kN - 1 - idx : idx;
                    const int b = idx & 1;
                    // buffer b last held agent idx - 2: its logits are read first
                    if (idx >= 2) consume(idx - 2);
                    if (mine) {
                        float o[kObsPad];
                        spread_obs_dyn<kN, kObsPad>(s, k, o);
                        float4* orow = reinterpret_cast<float4*>(a.obs + (ix + k) * kObsPad);
#pragma unroll
                        for (int q = 0; q < kObsPad / 4; ++q)
                            orow[q] = make_float4(o[4 * q], o[4 * q + 1], o[4 * q + 2], o[4 * q + 3]);
                        uint32_t w[kK1 / 2];
#pragma unroll
                        for (int i = 0; i < kK1 / 2; ++i)
                            w[i] = 2 * i + 1 < kObs ? tc::pack_bf16(o[2 * i], o[2 * i + 1]) : 0u;
                        uint8_t* xt = smem + kX + (g * 2 + b) * Eng::kXBytes;
#pragma unroll
                        for (int c = 0; c < kK1 / 8; ++c)
                            *reinterpret_cast<uint4*>(xt + Eng::x_offset(e, 8 * c)) =
                                make_uint4(w[4 * c], w[4 * c + 1], w[4 * c + 2], w[4 * c + 3]);
                        fence_proxy_async_smem();
                    }
                    group_sync(g);                                  // tile written, old logits read
                    if (e == 0) mbar_arrive_release(&x_full[g][b]);
                }
                consume(kN - 2);
                consume(kN - 1);
                group_sync(g);                                      // every agent's actions stored
                if (mine) {
                    int act[kN];
#pragma unroll
                    for (int i = 0; i < kN; ++i) act[i] = ag[i * 128 + e];
                    float r[kN];
                    spread_step<kN, kContact>(s, act, r, a.local_ratio);
#pragma unroll
                    for (int i = 0; i < kN; ++i) a.reward[ix + i] = r[i];
                    a.done[(ep * T + t) * a.n_envs + env] = (t == T - 1) ? 1 : 0;
                }
            }
        }
    }
    tc::fence_before_sync();
    __syncthreads();
    if (warp == 0) tc::tmem_dealloc(tbase, Eng::kTmemCols);
}

}  // namespace

bool spread_tc_supported(int n_agents, int obs_dim, int n_actions, int64_t envs_per_pair) {
    return n_agents == kN && obs_dim == kObs && n_actions == kA && envs_per_pair >= 1 &&
           envs_per_pair <= 128;
}

template <bool kContact, bool kLogits>
cudaError_t launch_tc(const RolloutArgs& a, int n_sm, cudaStream_t s) {
    cudaError_t err = cudaFuncSetAttribute(spread_rollout_tc_kernel<kContact, kLogits>,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmem);
    if (err != cudaSuccess) return err;
    const int64_t items = (int64_t)a.n_pairs * a.n_episodes;
    const int64_t ctas = items < n_sm ? items : n_sm;
    spread_rollout_tc_kernel<kContact, kLogits><<<(unsigned)ctas, kThreads, kSmem, s>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_spread_rollout_tc(const RolloutArgs& a, int n_sm, cudaStream_t s) {
    if (a.n_pairs == 0 || a.n_episodes == 0) return cudaSuccess;
    if (a.logits)
        return a.contact ? launch_tc<true, true>(a, n_sm, s) : launch_tc<false, true>(a, n_sm, s);
    return a.contact ? launch_tc<true, false>(a, n_sm, s) : launch_tc<false, false>(a, n_sm, s);
}

}  // namespace malib
