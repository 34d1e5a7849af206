// Batched rollout of cooperative particle spread with bf16 MLP policies on the
// tensor cores (Sec. 3.1 rollout under a policy combination; App. B.1 simple
// spread), for N = 8 agents with 34-float observations and 34-256-256-5 MLPs.
//
// A cluster of 8 CTAs serves one combination (one block of 128 environments):
// CTA k keeps the policy of agent k resident in shared memory and every CTA
// keeps a replica of all 128 environments' state in registers (one thread per
// environment). Per step, CTA k builds agent k's observations as a 128-row
// bf16 tile (the fp32 rows are staged in shared memory and leave as contiguous
// stores), runs it through the tensor-core MLP and draws agent k's actions.
// The 128 action bytes go to the 7 peers by asynchronous shared-memory stores
// that complete transaction counts on each peer's mbarrier, so a CTA waits
// only for the data it needs (bounded), with no cluster-wide barrier per step.
// Every CTA then applies the same 8 actions to its replica (identical IEEE
// operations, identical bits) and writes agent k's trajectory (observation,
// action, reward; CTA 0 the done flags).
#include "cluster.cuh"
#include "device_common.cuh"
#include "internal.h"
#include "mlp_tc.cuh"
#include "spread_env.cuh"

namespace malib {

namespace {

constexpr int kN = 8;                        // agents = landmarks = cluster size
constexpr int kObs = 34, kObsPad = 36, kK1 = 48, kA = 5;
using Eng = MlpTc<kK1, 256, 16, false>;      // biases read through L1 (shared memory is full)
constexpr int kThreads = 256;
constexpr uint32_t kX = Eng::kSmemBytes;                     // observation tile (bf16)
constexpr uint32_t kStage = kX + Eng::kXBytes;               // fp32 observation rows [128][36]
constexpr uint32_t kActs = kStage + 128 * kObsPad * 4;       // actions [parity][agent][env] u8
constexpr uint32_t kSmem = kActs + 2 * kN * 128;
static_assert(kX % 16 == 0 && kStage % 16 == 0 && kActs % 16 == 0, "16-byte aligned regions");
constexpr uint32_t kActTx = (kN - 1) * 128;                  // action bytes received per step

__device__ __forceinline__ void cluster_barrier_all() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n"
                 "barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

__global__ void __cluster_dims__(8, 1, 1) __launch_bounds__(kThreads, 1)
    spread_rollout_tc_kernel(RolloutArgs a) {
    extern __shared__ __align__(128) uint8_t smem[];
    __shared__ __align__(8) uint64_t stage_bar;
    __shared__ __align__(8) uint64_t mma_bar[2];
    __shared__ __align__(8) uint64_t act_bar[2];   // peers' actions of steps with parity 0 / 1
    __shared__ uint32_t tmem_base;

    uint8_t* acts = smem + kActs;
    const uint32_t me = cl::rank();
    const int tid = threadIdx.x, warp = tid >> 5;

    if (tid == 0) {
        mbar_init(&stage_bar, 1);
        mbar_init(&mma_bar[0], 1);
        mbar_init(&mma_bar[1], 1);
        mbar_init(&act_bar[0], 1);
        mbar_init(&act_bar[1], 1);
        mbar_arrive_expect_tx(&act_bar[0], kActTx);      // armed for steps 0 and 1
        mbar_arrive_expect_tx(&act_bar[1], kActTx);
    }
    if (warp == 0) {
        tc::tmem_alloc(&tmem_base, Eng::kTmemCols);
        tc::tmem_relinquish();
    }
    for (uint32_t i = tid * 16; i < Eng::kXBytes; i += kThreads * 16)
        *reinterpret_cast<uint4*>(smem + kX + i) = make_uint4(0, 0, 0, 0);
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    cluster_barrier_all();          // every peer's barriers exist before any remote store
    const uint32_t tbase = tmem_base;

    uint32_t stage_par = 0, mma_par = 0, step = 0;
    bool dead = false;              // a peer wait expired: stop waiting, results are flagged
    const int epp = (int)(a.n_envs / a.n_pairs);
    const int T = a.episode_len;
    const int64_t items = (int64_t)a.n_pairs * a.n_episodes;
    const int64_t n_cl = gridDim.x / kN, cid = blockIdx.x / kN;
    const int64_t per = (items + n_cl - 1) / n_cl;
    const int64_t lo = cid * per, hi = min(items, lo + per);
    int staged = -1;
    const float* gbias = nullptr;
    float* stage = reinterpret_cast<float*>(smem + kStage);

    for (int64_t it = lo; it < hi; ++it) {
        const int pair = (int)(it / a.n_episodes);
        const int64_t ep = it - (int64_t)pair * a.n_episodes;
        if (pair != staged) {
            bool ok = true;                  // every CTA checks all 8 ids: same decision
            for (int i = 0; i < kN; ++i) {
                const int p = a.pairs[pair * kN + i];
                ok = ok && p >= 0 && p < a.n_pol;
            }
            if (!ok) {
                if (tid == 0 && me == 0) atomicOr(a.err, ERRBIT_BAD_PAIR);
                continue;
            }
            __syncthreads();
            const float* policy = a.arena + a.pol_offset[a.pairs[pair * kN + me]];
            gbias = policy + Eng::kBias / 4;
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
            staged = pair;
            Eng::prefill_d1(smem, gbias, tbase);   // the new policy's b1 into D1 (ordered by
                                                   // the forward's opening hand-off)
        }

        const bool mine = tid < epp;
        const int64_t env = (int64_t)pair * epp + tid;
        const uint64_t g = (uint64_t)ep * (uint64_t)a.n_envs + (uint64_t)env;
        SpreadEnv<kN> s;
        if (mine) spread_reset<kN>(s, g, a.seed);

        for (int t = 0; t < T; ++t) {
            const uint32_t par = step & 1u;
            const int64_t ix = ((ep * T + t) * a.n_envs + env) * kN;
            uint8_t* my_acts = acts + (par * kN + me) * 128;
            float u = 0.f;
            if (mine) {
                u = u24(draw(g, (uint32_t)t, me, a.seed).x);      // ready before the logits
                float o[kObsPad];
                spread_obs_dyn<kN, kObsPad>(s, (int)me, o);
                float4* srow = reinterpret_cast<float4*>(stage + tid * kObsPad);
#pragma unroll
                for (int q = 0; q < kObsPad / 4; ++q)
                    srow[q] = make_float4(o[4 * q], o[4 * q + 1], o[4 * q + 2], o[4 * q + 3]);
                uint32_t w[kK1 / 2];
#pragma unroll
                for (int i = 0; i < kK1 / 2; ++i)
                    w[i] = 2 * i + 1 < kObs ? tc::pack_bf16(o[2 * i], o[2 * i + 1]) : 0u;
#pragma unroll
                for (int c = 0; c < kK1 / 8; ++c)
                    *reinterpret_cast<uint4*>(smem + kX + Eng::x_offset(tid, 8 * c)) =
                        make_uint4(w[4 * c], w[4 * c + 1], w[4 * c + 2], w[4 * c + 3]);
            }
            __syncthreads();
            {   // observations of agent me: [ep][t][env][agent][obs_pad], 144-byte runs per env
                const int64_t base = ((ep * T + t) * a.n_envs + (int64_t)pair * epp) * kN + me;
                const float4* src = reinterpret_cast<const float4*>(stage);
                for (int q = tid; q < epp * (kObsPad / 4); q += kThreads) {
                    const int v = q / (kObsPad / 4), c = q - v * (kObsPad / 4);
                    reinterpret_cast<float4*>(a.obs + (base + (int64_t)v * kN) * kObsPad)[c] = src[q];
                }
            }
            Eng::forward(smem, gbias, tbase, mma_bar, mma_par, a.err, [&](int row, const float* lg) {
                int act = 0;
                if (row < epp) {
                    float l5[kA];
#pragma unroll
                    for (int k = 0; k < kA; ++k) l5[k] = lg[k];
                    act = sample_masked<kA>(l5, 0x1Fu, u);
                    if (a.logits)
#pragma unroll
                        for (int k = 0; k < kA; ++k) a.logits[(ix + me) * kA + k] = l5[k];
                    a.action[ix + me] = (uint8_t)act;
                }
                my_acts[row] = (uint8_t)act;
            }, smem_u32(smem + kX));
            // forward ends with a CTA barrier: all 128 action bytes are in my_acts
            if (tid < (kN - 1) * 8) {
                const uint32_t c = (uint32_t)tid & 7u, j = (uint32_t)tid >> 3;
                const uint32_t r = j < me ? j : j + 1;
                const uint4 v = *reinterpret_cast<const uint4*>(my_acts + 16 * c);
                cl::st_async_v4(cl::map(my_acts + 16 * c, r), v, cl::map(&act_bar[par], r));
            }
            if (!dead && !cl::wait_cluster_bounded(&act_bar[par], (step >> 1) & 1u, kWaitLimitNs)) {
                dead = true;
                atomicOr(a.err, ERRBIT_TIMEOUT);
            }
            if (tid == 0) mbar_arrive_expect_tx(&act_bar[par], kActTx);   // re-armed for step + 2
            if (mine) {
                int act[kN];
#pragma unroll
                for (int i = 0; i < kN; ++i) act[i] = acts[(par * kN + i) * 128 + tid];
                float r[kN];
                spread_step<kN>(s, act, r, a.local_ratio);
                float rm = 0.f;
#pragma unroll
                for (int i = 0; i < kN; ++i)
                    if (i == (int)me) rm = r[i];
                a.reward[ix + me] = rm;
                if (me == 0) a.done[(ep * T + t) * a.n_envs + env] = (t == T - 1) ? 1 : 0;
            }
            ++step;
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
