// Batched rollout of the cooperative particle-spread scenario (App. B.1: N
// agents cover N landmarks; shared reward minus the summed distance from each
// landmark to its closest agent, minus one per collision) under policy
// combinations (Sec. 3.1: X ~ P(s, a, s' | a ~ Comb_t)), fp32 MLP policies.
//
// Work unit = (combination, episode pair): the combination's block of
// envs_per_pair (<= 128) environments for T steps, in two episodes at once.
// Each CTA takes a contiguous, equal-sized range of units (combination-major,
// so the N policies are staged into shared memory by bulk copy only when the
// combination changes). Thread t steps environment t % 128 of episode slot
// t / 128 with its state in registers; per step agent i's observations of both
// episodes form one 256-row pass of agent i's policy through the fp32 MLP
// engine. The observation tile is laid out [row][agent][obs_pad], the order of
// the trajectory, so each episode's observations of a step leave shared memory
// as one bulk copy; actions, rewards and done flags are stored per thread.
// The same kernel, templated on the scenario, runs the simple adversary, the
// simple speaker listener, the simple push, the simple tag and the simple
// reference (App. B.1) with their own environment code, and spread with contact
// forces between agents.
#include "adversary_env.cuh"
#include "push_env.cuh"
#include "ref_env.cuh"
#include "sl_env.cuh"
#include "tag_env.cuh"
#include "device_common.cuh"
#include "internal.h"
#include "mlp_f32.cuh"
#include "spread_env.cuh"

namespace malib {

namespace {

// Shared memory: the N policies, the observation tile X, layer 1's output H1
// and the logits LG. When the tiles of all N agents do not fit (the simple tag),
// the kernel runs per agent (kPerAgent): X and LG hold one agent's rows, each
// agent's observations are built just before its pass and stored to the
// trajectory from registers, and its action is drawn right after it.
template <int N, int IN, int H, int A = 5>
struct SpreadF32Smem {
    static_assert(H == 64, "the 256-row engine has 64 hidden units");
    using M = MlpF32R8<IN, A>;
    using L = F32Layout<IN, H, A>;
    static constexpr int R = M::kRows;            // 2 episode slots x 128 envs
    static constexpr size_t kAllBytes =
        (size_t)(N * L::kSize + N * R * M::XS + R * M::HS + N * R * M::LS) * 4;
    static constexpr bool kPerAgent = kAllBytes > 232448;
    static constexpr int kNX = kPerAgent ? 1 : N;   // agents' tiles held at once
    static constexpr int kW = 0;
    static constexpr int kX = kW + N * L::kSize;
    static constexpr int kH1 = kX + kNX * R * M::XS;
    static constexpr int kLG = kH1 + R * M::HS;
    static constexpr int kFloats = kLG + kNX * R * M::LS;
    static constexpr size_t kBytes = (size_t)kFloats * 4;
    static_assert(kBytes <= 232448, "fits the 227 KB of shared memory of a CTA");
};

// kScen: kSpread - cooperative spread (N agents, N landmarks); kAdversary - the
// simple adversary (N = 3, two landmarks, obs 14); kSpeakerListener - the simple
// speaker listener (N = 2, three landmarks, obs 11; the speaker may take
// actions 0..2 only); kPush - the simple push (N = 2, one landmark, obs 8);
// kTag - the simple tag (N = 4, two obstacles, obs 16); kSpreadContact -
// spread whose agents also push each other apart; kReference - the simple
// reference (N = 2, three landmarks, obs 14, 15 actions: move and message).
constexpr int kSpread = 0, kAdversary = 1, kSpeakerListener = 2, kPush = 3, kTag = 4, kSpreadContact = 5,
              kReference = 6;
__host__ __device__ constexpr int actions_of(int scen) { return scen == kReference ? kRefActions : 5; }

template <int kScen, int N>
struct ScenarioEnv {
    using type = SpreadEnv<N>;
};
template <int N>
struct ScenarioEnv<kAdversary, N> {
    using type = AdvEnv;
};
template <int N>
struct ScenarioEnv<kSpeakerListener, N> {
    using type = SlEnv;
};
template <int N>
struct ScenarioEnv<kPush, N> {
    using type = PushEnv;
};
template <int N>
struct ScenarioEnv<kTag, N> {
    using type = TagEnv;
};
template <int N>
struct ScenarioEnv<kReference, N> {
    using type = RefEnv;
};

// kLogits: the call records the logits (the recording code is compiled out of
// the other instance).
template <int N, int IN, int H, int kScen = kSpread, bool kLogits = false>
__global__ void __launch_bounds__(256, 1) spread_rollout_f32_kernel(RolloutArgs a) {
    static_assert(kScen != kAdversary || (N == 3 && IN == kAdvObs), "the simple adversary has 3 agents, obs 14");
    static_assert(kScen != kSpeakerListener || (N == 2 && IN == kSlObs),
                  "the simple speaker listener has 2 agents, obs 11");
    static_assert(kScen != kPush || (N == 2 && IN == kPushObs), "the simple push has 2 agents, obs 8");
    static_assert(kScen != kTag || (N == 4 && IN == kTagObs), "the simple tag has 4 agents, obs 16");
    static_assert(kScen != kReference || (N == 2 && IN == kRefObs), "the simple reference has 2 agents, obs 14");
    constexpr int A = actions_of(kScen);
    using SM = SpreadF32Smem<N, IN, H, A>;
    using M = typename SM::M;
    using L = typename SM::L;
    constexpr int R = SM::R;
    constexpr int XS = M::XS;           // == obs_pad
    extern __shared__ __align__(128) float smem[];
    float* Ws = smem + SM::kW;
    float* X = smem + SM::kX;
    float* H1 = smem + SM::kH1;
    float* LG = smem + SM::kLG;
    __shared__ __align__(8) uint64_t bar;

    const int tid = threadIdx.x;
    const int slot = tid >> 7, v = tid & 127;        // episode slot, env of the combination
    for (int i = tid; i < R * SM::kNX * XS; i += blockDim.x) X[i] = 0.f;
    if (tid == 0) mbar_init(&bar, 1);
    __syncthreads();
    uint32_t parity = 0;

    const int epp = (int)(a.n_envs / a.n_pairs);
    const int T = a.episode_len;
    const int64_t upp = (a.n_episodes + 1) / 2;         // units (episode pairs) per combination
    const int64_t units = (int64_t)a.n_pairs * upp;
    const int64_t lo = units * blockIdx.x / gridDim.x;
    const int64_t hi = units * (blockIdx.x + 1) / gridDim.x;
    int staged = -1;

    for (int64_t u = lo; u < hi; ++u) {
        const int pair = (int)(u / upp);
        const int64_t ep0 = 2 * (u - (int64_t)pair * upp);
        if (pair != staged) {
            bool ok = true;
            for (int i = 0; i < N; ++i) {
                const int p = a.pairs[pair * N + i];
                ok = ok && p >= 0 && p < a.n_pol;
            }
            if (!ok) {
                if (tid == 0) atomicOr(a.err, ERRBIT_BAD_PAIR);
                continue;
            }
            __syncthreads();   // everyone is done with the previous weights
            if (tid == 0) {
                fence_proxy_async_smem();
                mbar_arrive_expect_tx(&bar, (uint32_t)N * L::kSize * 4u);
                for (int i = 0; i < N; ++i)
                    bulk_g2s(Ws + i * L::kSize, a.arena + a.pol_offset[a.pairs[pair * N + i]],
                             (uint32_t)L::kSize * 4u, &bar);
            }
            if (!mbar_wait_bounded(&bar, parity, kWaitLimitNs)) {
                if (tid == 0) {
                    atomicOr(a.err, ERRBIT_TIMEOUT);
                    bulk_wait_all();
                }
                mbar_wait_bounded(&bar, parity, kWaitLimitNs);
                return;
            }
            parity ^= 1u;
            staged = pair;
        }

        const int64_t ep = ep0 + slot;
        const int n_slots = ep0 + 1 < a.n_episodes ? 2 : 1;
        const bool mine = slot < n_slots && v < epp;
        const int64_t env = (int64_t)pair * epp + v;
        const uint64_t g = (uint64_t)ep * (uint64_t)a.n_envs + (uint64_t)env;
        typename ScenarioEnv<kScen, N>::type s;
        if (mine) {
            if constexpr (kScen == kAdversary) adv_reset(s, g, a.seed);
            else if constexpr (kScen == kSpeakerListener) sl_reset(s, g, a.seed);
            else if constexpr (kScen == kPush) push_reset(s, g, a.seed);
            else if constexpr (kScen == kTag) tag_reset(s, g, a.seed);
            else if constexpr (kScen == kReference) ref_reset(s, g, a.seed);
            else spread_reset<N>(s, g, a.seed);
        }

        for (int t = 0; t < T; ++t) {
            if constexpr (SM::kPerAgent) {
                // one agent at a time: its observations (to X and the
                // trajectory), its pass, its draw. The loop stays rolled, so the
                // MLP's code appears once (instruction fetch limited the unrolled
                // form); the observation is built by a copy per constant agent
                // index (no dynamic indexing of the state in registers), and the
                // actions are packed one byte per agent.
                static_assert(N <= 4, "one byte per agent's action in a 32-bit word");
                uint32_t act_pk = 0;
                const int64_t ix = ((ep * T + t) * a.n_envs + env) * N;
#pragma unroll 1
                for (int i = 0; i < N; ++i) {
                    if (mine) {
                        float o[XS];
#pragma unroll
                        for (int j = 0; j < N; ++j) {
                            if (j != i) continue;
                            if constexpr (kScen == kTag) tag_obs<XS>(s, j, o);
                            else if constexpr (kScen == kReference) ref_obs<XS>(s, j, o);
                            else if constexpr (kScen == kPush) push_obs<XS>(s, j, o);
                            else if constexpr (kScen == kAdversary) adv_obs<XS>(s, j, o);
                            else if constexpr (kScen == kSpeakerListener) sl_obs<XS>(s, j, o);
                            else spread_obs<N, XS>(s, j, o);
                        }
                        float4* xr = reinterpret_cast<float4*>(X + tid * XS);
                        float4* gr = reinterpret_cast<float4*>(a.obs + (ix + i) * XS);
#pragma unroll
                        for (int q = 0; q < XS / 4; ++q) {
                            const float4 f = make_float4(o[4 * q], o[4 * q + 1], o[4 * q + 2], o[4 * q + 3]);
                            xr[q] = f;
                            gr[q] = f;
                        }
                    }
                    __syncthreads();
                    const float* w = Ws + i * L::kSize;
                    M::template layer1<XS>(X, H1, w + L::kW1T, w + L::kB1);
                    M::layer23(H1, LG, w + L::kW2T, w + L::kB2, w + L::kW3, w + L::kB3);
                    if (mine) {
                        // LG is rewritten only after the next pass's layer-1 barrier
                        float lg[A];
#pragma unroll
                        for (int k = 0; k < A; ++k) lg[k] = LG[tid * M::LS + k];
                        const float uu = u24(draw(g, (uint32_t)t, (uint32_t)i, a.seed).x);
                        const unsigned legal = (kScen == kSpeakerListener && i == 0) ? kSlSpeakerLegal : (1u << A) - 1u;
                        act_pk |= (uint32_t)sample_masked<A>(lg, legal, uu) << (8 * i);
                        if (kLogits)
#pragma unroll
                            for (int k = 0; k < A; ++k) a.logits[(ix + i) * A + k] = lg[k];
                    }
                }
                if (mine) {
                    int act[N];
#pragma unroll
                    for (int i = 0; i < N; ++i) act[i] = (int)((act_pk >> (8 * i)) & 0xffu);
                    float r[N];
                    if constexpr (kScen == kAdversary) adv_step(s, act, r);
                    else if constexpr (kScen == kSpeakerListener) sl_step(s, act, r);
                    else if constexpr (kScen == kPush) push_step(s, act, r);
                    else if constexpr (kScen == kTag) tag_step(s, act, r);
                    else if constexpr (kScen == kReference) ref_step(s, act, r, a.local_ratio < 0.f ? 0.5f : a.local_ratio);
                    else spread_step<N, kScen == kSpreadContact>(s, act, r, a.local_ratio);
#pragma unroll
                    for (int i = 0; i < N; ++i) {
                        a.action[ix + i] = (uint8_t)act[i];
                        a.reward[ix + i] = r[i];
                    }
                    a.done[(ep * T + t) * a.n_envs + env] = (t == T - 1) ? 1 : 0;
                }
                continue;
            }
            if (mine) {
#pragma unroll
                for (int i = 0; i < N; ++i) {
                    float o[XS];
                    if constexpr (kScen == kAdversary) adv_obs<XS>(s, i, o);
                    else if constexpr (kScen == kSpeakerListener) sl_obs<XS>(s, i, o);
                    else if constexpr (kScen == kPush) push_obs<XS>(s, i, o);
                    else if constexpr (kScen == kTag) tag_obs<XS>(s, i, o);
                    else if constexpr (kScen == kReference) ref_obs<XS>(s, i, o);
                    else spread_obs<N, XS>(s, i, o);
                    float4* xr = reinterpret_cast<float4*>(X + (tid * N + i) * XS);
#pragma unroll
                    for (int q = 0; q < XS / 4; ++q)
                        xr[q] = make_float4(o[4 * q], o[4 * q + 1], o[4 * q + 2], o[4 * q + 3]);
                }
                fence_proxy_async_smem();                // the rows are read by bulk copies
            }
            __syncthreads();
            // trajectory observations, [ep][t][env][agent][XS]: an episode's rows
            // are contiguous in the tile and in the trajectory
            if (tid == 0) {
                for (int sl = 0; sl < n_slots; ++sl) {
                    const int64_t row_base = (((ep0 + sl) * T + t) * a.n_envs + (int64_t)pair * epp) * N;
                    bulk_s2g(a.obs + row_base * XS, X + sl * 128 * N * XS, (uint32_t)(epp * N * XS * 4));
                }
                bulk_commit();
            }
            for (int i = 0; i < N; ++i) {
                const float* w = Ws + i * L::kSize;
                M::template layer1<N * XS>(X + i * XS, H1, w + L::kW1T, w + L::kB1);
                // the copies have read the tile before the last pass's barrier;
                // the tile is rewritten only after it
                if (i == N - 1 && tid == 0) bulk_wait_read();
                M::layer23(H1, LG + i * R * M::LS, w + L::kW2T, w + L::kB2, w + L::kW3, w + L::kB3);
            }
            if (mine) {
                int act[N];
                float r[N];
                const int64_t ix = ((ep * T + t) * a.n_envs + env) * N;
#pragma unroll
                for (int i = 0; i < N; ++i) {
                    float lg[A];
#pragma unroll
                    for (int k = 0; k < A; ++k) lg[k] = LG[(i * R + tid) * M::LS + k];
                    const float uu = u24(draw(g, (uint32_t)t, (uint32_t)i, a.seed).x);
                    const unsigned legal = (kScen == kSpeakerListener && i == 0) ? kSlSpeakerLegal : (1u << A) - 1u;
                    act[i] = sample_masked<A>(lg, legal, uu);
                    if (kLogits)
#pragma unroll
                        for (int k = 0; k < A; ++k) a.logits[(ix + i) * A + k] = lg[k];
                }
                if constexpr (kScen == kAdversary) adv_step(s, act, r);
                else if constexpr (kScen == kSpeakerListener) sl_step(s, act, r);
                else if constexpr (kScen == kPush) push_step(s, act, r);
                else if constexpr (kScen == kTag) tag_step(s, act, r);
                else if constexpr (kScen == kReference) ref_step(s, act, r, a.local_ratio < 0.f ? 0.5f : a.local_ratio);
                else spread_step<N, kScen == kSpreadContact>(s, act, r, a.local_ratio);
#pragma unroll
                for (int i = 0; i < N; ++i) {
                    a.action[ix + i] = (uint8_t)act[i];
                    a.reward[ix + i] = r[i];
                }
                a.done[(ep * T + t) * a.n_envs + env] = (t == T - 1) ? 1 : 0;
            }
            // X is rewritten next step only after the passes' trailing barrier;
            // LG is rewritten only after next step's first barrier.
        }
    }
    if (tid == 0) bulk_wait_all();   // the trajectory copies have landed
}

template <int N, int IN, int H, int kScen = kSpread>
cudaError_t launch_spread_nih(const RolloutArgs& a, int n_sm, cudaStream_t s) {
    using SM = SpreadF32Smem<N, IN, H, actions_of(kScen)>;
    auto kern = a.logits ? spread_rollout_f32_kernel<N, IN, H, kScen, true>
                         : spread_rollout_f32_kernel<N, IN, H, kScen, false>;
    cudaError_t err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)SM::kBytes);
    if (err != cudaSuccess) return err;
    const int64_t units = (int64_t)a.n_pairs * ((a.n_episodes + 1) / 2);
    int64_t grid = units < n_sm ? units : n_sm;
    if (grid < 1) grid = 1;
    kern<<<(unsigned)grid, 256, SM::kBytes, s>>>(a);
    return cudaGetLastError();
}

}  // namespace

bool scenario_f32_supported(int hidden) { return hidden == 64; }

bool spread_f32_supported(int n_agents, int obs_dim, int hidden) {
    return n_agents == 3 && obs_dim == 18 && hidden == 64;
}

cudaError_t launch_spread_rollout_f32(const RolloutArgs& a, int hidden, int n_sm, cudaStream_t s) {
    if (a.n_pairs == 0 || a.n_episodes == 0) return cudaSuccess;
    if (a.env_kind == MALIB_ENV_ADVERSARY) {
        if (hidden == 64) return launch_spread_nih<3, kAdvObs, 64, kAdversary>(a, n_sm, s);
        return cudaErrorInvalidValue;
    }
    if (a.env_kind == MALIB_ENV_SPEAKER_LISTENER) {
        if (hidden == 64) return launch_spread_nih<2, kSlObs, 64, kSpeakerListener>(a, n_sm, s);
        return cudaErrorInvalidValue;
    }
    if (a.env_kind == MALIB_ENV_PUSH) {
        if (hidden == 64) return launch_spread_nih<2, kPushObs, 64, kPush>(a, n_sm, s);
        return cudaErrorInvalidValue;
    }
    if (a.env_kind == MALIB_ENV_REFERENCE) {
        if (hidden == 64) return launch_spread_nih<2, kRefObs, 64, kReference>(a, n_sm, s);
        return cudaErrorInvalidValue;
    }
    if (a.env_kind == MALIB_ENV_TAG) {
        if (hidden == 64) return launch_spread_nih<4, kTagObs, 64, kTag>(a, n_sm, s);
        return cudaErrorInvalidValue;
    }
    if (a.n_agents == 3 && a.obs_dim == 18 && hidden == 64)
        return a.contact ? launch_spread_nih<3, 18, 64, kSpreadContact>(a, n_sm, s)
                         : launch_spread_nih<3, 18, 64>(a, n_sm, s);
    return cudaErrorInvalidValue;
}

}  // namespace malib
