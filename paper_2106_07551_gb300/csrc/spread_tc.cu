// Batched rollout of cooperative particle spread with bf16 MLP policies on the
// tensor cores (Sec. 3.1 rollout under a policy combination; App. B.1 simple
// spread), for N = 8 agents with 34-float observations and 34-256-256-5 MLPs.
//
// A cluster of 8 CTAs serves one combination (one block of 128 environments):
// CTA k keeps the policy of agent k resident in shared memory. Each CTA has 16
// warps in three roles:
//  * warps 0-7, the engine: runs agent k's 128-row observation tiles through
//    the tensor-core MLP (hidden activations in tensor memory) and hands the
//    logits to the tile's group through shared memory and a local mbarrier;
//  * warps 8-11 and 12-15, environment groups 0 and 1: two episodes of the
//    combination in flight, one environment per thread. Every CTA keeps a
//    replica of a group's 128 environments; per step a group builds agent k's
//    observations (a bf16 tile for the engine; each thread stores its fp32 row,
//    one 144-byte run, to the trajectory), draws agent k's actions from the
//    engine's logits and sends them to all 8 CTAs, waits for the 8 agents'
//    actions, applies them
//    (identical IEEE operations in every CTA, identical bits) and writes agent
//    k's trajectory (observation, action, reward; CTA 0 the done flags).
// While the engine runs one group's tile, the other group steps its
// environments, so the environment work overlaps the forward. Actions travel
// as asynchronous stores into every CTA's shared memory (this one included)
// that complete transaction bytes on the receiving group's per-parity
// mbarrier (1,024 bytes expected per step); a group's tile is handed to the
// engine through a local mbarrier. Every wait is bounded.
#include "cluster.cuh"
#include "device_common.cuh"
#include "internal.h"
#include "mlp_tc.cuh"
#include "spread_env.cuh"

namespace malib {

namespace {

constexpr int kN = 8;                        // agents = landmarks = cluster size
constexpr int kObs = 34, kObsPad = 36, kK1 = 48, kA = 5;
using Eng = MlpTc<kK1, 256, 16, true, /*kBarId=*/1>;    // biases staged with the weights
constexpr int kThreads = 512;
constexpr int kEngineThreads = 256;
constexpr int kGroups = 2;
constexpr uint32_t kX = Eng::kSmemBytes;                          // observation tiles [group]
constexpr uint32_t kActs = kX + kGroups * Eng::kXBytes;           // [group][parity][agent][env]
constexpr uint32_t kSend = kActs + kGroups * 2 * kN * 128;        // this agent's actions [group][env]
constexpr uint32_t kLgs = kSend + kGroups * 128;                  // logits [group][env][8] fp32
constexpr uint32_t kSmem = kLgs + kGroups * 128 * 8 * 4;
static_assert(kX % 16 == 0 && kActs % 16 == 0 && kSend % 16 == 0 &&
              kLgs % 16 == 0, "16-byte aligned regions");
constexpr uint32_t kActTx = kN * 128;                             // action bytes received per step

__device__ __forceinline__ void cluster_barrier_all() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n"
                 "barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

__device__ __forceinline__ void group_sync(int g) {
    if (g == 0) asm volatile("bar.sync 2, 128;" ::: "memory");
    else asm volatile("bar.sync 3, 128;" ::: "memory");
}

// The items of a cluster, (combination, episode) pairs in order, are taken two
// at a time: group 0 the first, group 1 the next one when it belongs to the
// same combination (else group 1 idles that round). Every role of every CTA
// walks the same rounds.
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
    bool ok = true;                  // every CTA checks all 8 ids: same decision
    for (int i = 0; i < kN; ++i) {
        const int p = a.pairs[pair * kN + i];
        ok = ok && p >= 0 && p < a.n_pol;
    }
    return ok;
}

__global__ void __cluster_dims__(8, 1, 1) __launch_bounds__(kThreads, 1)
    spread_rollout_tc_kernel(RolloutArgs a) {
    extern __shared__ __align__(128) uint8_t smem[];
    __shared__ __align__(8) uint64_t stage_bar;
    __shared__ __align__(8) uint64_t mma_bar[2];
    __shared__ __align__(8) uint64_t act_bar[kGroups][2];   // actions of a group's steps, by parity
    __shared__ __align__(8) uint64_t x_bar[kGroups];        // a group's tile is ready
    __shared__ __align__(8) uint64_t lg_bar[kGroups];       // a group's logits are ready
    __shared__ uint32_t tmem_base;

    uint8_t* acts = smem + kActs;
    uint8_t* send = smem + kSend;
    float* lgs = reinterpret_cast<float*>(smem + kLgs);
    const uint32_t me = cl::rank();
    const int tid = threadIdx.x, warp = tid >> 5;

    if (tid == 0) {
        mbar_init(&stage_bar, 1);
        mbar_init(&mma_bar[0], 1);
        mbar_init(&mma_bar[1], 1);
        for (int g = 0; g < kGroups; ++g) {
            mbar_init(&x_bar[g], 1);
            mbar_init(&lg_bar[g], 1);
            for (int p = 0; p < 2; ++p) {
                mbar_init(&act_bar[g][p], 1);
                mbar_arrive_expect_tx(&act_bar[g][p], kActTx);   // armed for steps 0 and 1
            }
        }
    }
    if (warp == 0) {
        tc::tmem_alloc(&tmem_base, Eng::kTmemCols);
        tc::tmem_relinquish();
    }
    for (uint32_t i = tid * 16; i < kGroups * Eng::kXBytes; i += kThreads * 16)
        *reinterpret_cast<uint4*>(smem + kX + i) = make_uint4(0, 0, 0, 0);
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    cluster_barrier_all();          // every peer's barriers exist before any remote store
    const uint32_t tbase = tmem_base;

    const int epp = (int)(a.n_envs / a.n_pairs);
    const int T = a.episode_len;
    const int64_t items = (int64_t)a.n_pairs * a.n_episodes;
    const int64_t n_cl = gridDim.x / kN, cid = blockIdx.x / kN;
    const int64_t per = (items + n_cl - 1) / n_cl;
    const int64_t lo = cid * per, hi = min(items, lo + per);

    if (warp < 8) {
        // ------------------------------------------------------------ engine
        uint32_t stage_par = 0, mma_par = 0, x_bits = 0;
        int staged = -1;
        for (int64_t it = lo; it < hi;) {
            const Round rd = round_at(it, hi, a.n_episodes);
            it = rd.next;
            if (!pair_valid(a, rd.pair)) {
                if (tid == 0 && me == 0) atomicOr(a.err, ERRBIT_BAD_PAIR);
                continue;
            }
            if (rd.pair != staged) {
                const float* policy = a.arena + a.pol_offset[a.pairs[rd.pair * kN + me]];
                Eng::sync();                 // the previous forwards are complete
                if (tid == 0) {
                    fence_proxy_async_smem();
                    mbar_arrive_expect_tx(&stage_bar, Eng::kStageBytes);
                    for (uint32_t off = 0; off < Eng::kStageBytes; off += 32768u)
                        bulk_g2s(smem + off, reinterpret_cast<const uint8_t*>(policy) + off,
                                 min(32768u, Eng::kStageBytes - off), &stage_bar);
                }
                if (!mbar_wait_bounded(&stage_bar, stage_par, kWaitLimitNs) && tid == 0)
                    atomicOr(a.err, ERRBIT_TIMEOUT);
                stage_par ^= 1u;
                staged = rd.pair;
                tc::fence_before_sync();
                Eng::sync();
            }
            for (int t = 0; t < T; ++t) {
                for (int g = 0; g < kGroups; ++g) {
                    if (rd.ep[g] < 0) continue;
                    if (tid == 0 &&
                        !mbar_wait_bounded(&x_bar[g], (x_bits >> g) & 1u, kWaitLimitNs))
                        atomicOr(a.err, ERRBIT_TIMEOUT);
                    x_bits ^= 1u << g;
                    Eng::sync();
                    float* lgg = lgs + g * 128 * 8;
                    Eng::forward(smem, nullptr, tbase, mma_bar, mma_par, a.err,
                                 [&](int row, const float* lg) {
                                     float4* d = reinterpret_cast<float4*>(lgg + row * 8);
                                     d[0] = make_float4(lg[0], lg[1], lg[2], lg[3]);
                                     d[1] = make_float4(lg[4], 0.f, 0.f, 0.f);
                                 },
                                 smem_u32(smem + kX + g * Eng::kXBytes), /*x_published=*/true);
                    // the forward ends with an engine barrier: every row's logits are stored
                    if (tid == 0) mbar_arrive_release(&lg_bar[g]);
                }
            }
        }
    } else {
        // ------------------------------------------------------------ environment groups
        const int g = (warp - 8) >> 2;
        const int e = tid - kEngineThreads - g * 128;     // environment within the block
        uint8_t* xg = smem + kX + g * Eng::kXBytes;
        uint32_t act_bits = 0;                             // act_bar[g][p] phase: bit p
        uint32_t lg_par = 0;
        const float* lgg = lgs + g * 128 * 8;
        uint8_t* snd = send + g * 128;
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
                const uint32_t par = (uint32_t)t & 1u;
                float u = 0.f;
                if (mine) {
                    u = u24(draw(gid, (uint32_t)t, me, a.seed).x);
                    float o[kObsPad];
                    spread_obs_dyn<kN, kObsPad>(s, (int)me, o);
                    // agent me's observation: [ep][t][env][agent][obs_pad], one 144-byte run
                    float4* orow = reinterpret_cast<float4*>(
                        a.obs + (((ep * T + t) * a.n_envs + env) * kN + me) * kObsPad);
#pragma unroll
                    for (int q = 0; q < kObsPad / 4; ++q)
                        orow[q] = make_float4(o[4 * q], o[4 * q + 1], o[4 * q + 2], o[4 * q + 3]);
                    uint32_t w[kK1 / 2];
#pragma unroll
                    for (int i = 0; i < kK1 / 2; ++i)
                        w[i] = 2 * i + 1 < kObs ? tc::pack_bf16(o[2 * i], o[2 * i + 1]) : 0u;
#pragma unroll
                    for (int c = 0; c < kK1 / 8; ++c)
                        *reinterpret_cast<uint4*>(xg + Eng::x_offset(e, 8 * c)) =
                            make_uint4(w[4 * c], w[4 * c + 1], w[4 * c + 2], w[4 * c + 3]);
                    fence_proxy_async_smem();
                }
                group_sync(g);
                if (e == 0) mbar_arrive_release(&x_bar[g]);      // the tile goes to the engine
                // agent me's logits from the engine; its actions to every CTA
                if (!mbar_wait_bounded(&lg_bar[g], lg_par, kWaitLimitNs) && e == 0)
                    atomicOr(a.err, ERRBIT_TIMEOUT);
                lg_par ^= 1u;
                {
                    int act = 0;
                    if (mine) {
                        const float4 l0 = *reinterpret_cast<const float4*>(lgg + e * 8);
                        float l5[kA] = {l0.x, l0.y, l0.z, l0.w, lgg[e * 8 + 4]};
                        act = sample_masked<kA>(l5, 0x1Fu, u);
                        const int64_t ix = ((ep * T + t) * a.n_envs + env) * kN;
                        if (a.logits)
#pragma unroll
                            for (int k = 0; k < kA; ++k) a.logits[(ix + me) * kA + k] = l5[k];
                        a.action[ix + me] = (uint8_t)act;
                    }
                    snd[e] = (uint8_t)act;
                }
                group_sync(g);
                if (e < kN * 8) {
                    const uint32_t c = (uint32_t)e & 7u, r = (uint32_t)e >> 3;
                    uint8_t* dst = acts + ((g * 2 + par) * kN + me) * 128 + 16 * c;
                    cl::st_async_v4(cl::map(dst, r), *reinterpret_cast<const uint4*>(snd + 16 * c),
                                    cl::map(&act_bar[g][par], r));
                }
                // the 8 agents' actions of this step, from every engine of the cluster
                if (!cl::wait_cluster_bounded(&act_bar[g][par], (act_bits >> par) & 1u, kWaitLimitNs) &&
                    e == 0)
                    atomicOr(a.err, ERRBIT_TIMEOUT);
                act_bits ^= 1u << par;
                group_sync(g);                                  // every thread has seen the phase
                if (e == 0) mbar_arrive_expect_tx(&act_bar[g][par], kActTx);   // armed for t + 2
                if (mine) {
                    int act[kN];
#pragma unroll
                    for (int i = 0; i < kN; ++i) act[i] = acts[((g * 2 + par) * kN + i) * 128 + e];
                    float r[kN];
                    spread_step<kN>(s, act, r, a.local_ratio);
                    float rm = 0.f;
#pragma unroll
                    for (int i = 0; i < kN; ++i)
                        if (i == (int)me) rm = r[i];
                    const int64_t ix = ((ep * T + t) * a.n_envs + env) * kN;
                    a.reward[ix + me] = rm;
                    if (me == 0) a.done[(ep * T + t) * a.n_envs + env] = (t == T - 1) ? 1 : 0;
                }
                group_sync(g);       // the tile is rewritten next step
            }
        }
    }
    tc::fence_before_sync();
    __syncthreads();
    cluster_barrier_all();          // every remote store to this CTA was awaited before this
    if (warp == 0) tc::tmem_dealloc(tbase, Eng::kTmemCols);
}

}  // namespace

bool spread_tc_supported(int n_agents, int obs_dim, int n_actions, int64_t envs_per_pair) {
    return n_agents == kN && obs_dim == kObs && n_actions == kA && envs_per_pair >= 1 &&
           envs_per_pair <= 128;
}

cudaError_t launch_spread_rollout_tc(const RolloutArgs& a, int n_sm, cudaStream_t s) {
    if (a.n_pairs == 0 || a.n_episodes == 0) return cudaSuccess;
    cudaError_t err = cudaFuncSetAttribute(spread_rollout_tc_kernel,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmem);
    if (err != cudaSuccess) return err;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(kN, 1, 1);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = kSmem;
    cfg.stream = s;
    int max_clusters = 0;
    if (cudaOccupancyMaxActiveClusters(&max_clusters, spread_rollout_tc_kernel, &cfg) != cudaSuccess ||
        max_clusters < 1) {
        cudaGetLastError();
        max_clusters = n_sm / kN;
    }
    const int64_t items = (int64_t)a.n_pairs * a.n_episodes;
    int64_t clusters = items < max_clusters ? items : max_clusters;
    if (clusters < 1) clusters = 1;
    spread_rollout_tc_kernel<<<(unsigned)(kN * clusters), kThreads, kSmem, s>>>(a);
    return cudaGetLastError();
}

}  // namespace malib
