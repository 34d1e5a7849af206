// Payoff-table evaluation of Leduc hold'em with bf16 MLP policies on the
// tensor cores (Sec. 3.2 payoff table, Sec. 4.2 Monte-Carlo simulations per
// policy combination).
//
// A cluster of two CTAs evaluates one pair at a time. CTA r keeps the policy of
// seat r resident in shared memory (bf16 weight image and biases, ~157 KB) and
// owns 128 hands in flight. Rows 64 s .. 64 s + 63 of each CTA's 128-row tile
// belong to the hands of CTA s. Each step, the hands of a CTA are ranked by
// acting seat with warp ballots; the first 64 acting as seat r write their bf16
// observation into rows of CTA r's tile (the rest wait a step: a hand's
// randomness depends only on its own ids, so deferral changes no result). Each
// CTA runs its tile through the tensor-core MLP and returns every row's logits
// to the row's CTA. Both directions use asynchronous stores into the peer's
// shared memory that complete transaction counts on the receiver's mbarrier:
// every slot is written each step (unused rows with zeros) plus a 16-byte
// header (rows placed, live hands), so each receiver expects a fixed byte
// count and waits (bounded) for its data alone. Both CTAs take the same pair
// segments and leave a segment together, when neither holds a live hand.
#include "cluster.cuh"
#include "device_common.cuh"
#include "eval_common.cuh"
#include "internal.h"
#include "leduc_env.cuh"
#include "mlp_tc.cuh"

namespace malib {

namespace {

using Eng = MlpTc<32, 256, 16>;
constexpr int kSlots = 128;               // hands per CTA
constexpr int kPart = 64;                 // tile rows per source CTA
constexpr int kThreads = 256;
constexpr uint32_t kLg = Eng::kSmemBytes;                 // logits [target][rank][4] fp32
constexpr uint32_t kSmem = kLg + 2 * kPart * 16;
constexpr uint32_t kXTx = 2 * (kPart * 64 + 16);          // tile bytes + headers received per step
constexpr uint32_t kLgTx = 2 * kPart * 16;                // logits bytes received per step
constexpr int kMaxDec = 8;

__device__ __forceinline__ void cluster_barrier_all() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n"
                 "barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
    leduc_eval_tc_kernel(EvalArgs a) {
    extern __shared__ __align__(128) uint8_t smem[];
    __shared__ __align__(8) uint64_t stage_bar;
    __shared__ __align__(8) uint64_t mma_bar;
    __shared__ uint32_t tmem_base;
    __shared__ __align__(8) uint64_t x_bar;        // tile rows and headers of this step
    __shared__ __align__(8) uint64_t lg_bar;       // logits of this step
    __shared__ __align__(16) uint4 hdr[2];         // from CTA s: {rows placed here, live hands}
    __shared__ uint32_t dead_s, go_s;              // a peer wait expired; this step runs
    __shared__ int wcnt[2][8];
    __shared__ unsigned long long next_k;

    float* lgbuf = reinterpret_cast<float*>(smem + kLg);
    const uint32_t me = cl::rank();
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

    if (tid == 0) {
        mbar_init(&stage_bar, 1);
        mbar_init(&mma_bar, 1);
        dead_s = 0u;
        mbar_init(&x_bar, 1);
        mbar_init(&lg_bar, 1);
        mbar_arrive_expect_tx(&x_bar, kXTx);       // armed for the first step
        mbar_arrive_expect_tx(&lg_bar, kLgTx);
    }
    if (warp == 0) {
        tc::tmem_alloc(&tmem_base, Eng::kTmemCols);
        tc::tmem_relinquish();
    }
    for (uint32_t i = tid * 16; i < Eng::kActBytes; i += kThreads * 16)
        *reinterpret_cast<uint4*>(smem + Eng::kAct + i) = make_uint4(0, 0, 0, 0);
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    cluster_barrier_all();          // peers' barriers exist before any remote store
    const uint32_t tbase = tmem_base;

    uint32_t stage_par = 0, mma_par = 0, x_par = 0, lg_par = 0, step = 0;

    const int64_t total = (int64_t)a.n_pairs * a.n_episodes;
    const int64_t n_cl = gridDim.x / 2, cid = blockIdx.x / 2;
    const int64_t per = (total + n_cl - 1) / n_cl;
    const int64_t lo = cid * per, hi = min(total, lo + per);

    for (int64_t seg = lo; seg < hi;) {
        const int pair = (int)(seg / a.n_episodes);
        const int64_t e_lo = seg - (int64_t)pair * a.n_episodes;
        const int64_t e_hi = min(a.n_episodes, e_lo + (hi - seg));
        seg += e_hi - e_lo;
        const int p0 = a.pairs[2 * pair], p1 = a.pairs[2 * pair + 1];
        if (!pair_ok(a, p0, p1)) {          // same decision in both CTAs
            if (tid == 0 && me == 0) atomicOr(a.err, ERRBIT_BAD_PAIR);
            continue;
        }
        const float* policy = a.arena + a.pol_offset[me == 0 ? p0 : p1];
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

        // this CTA's hands: e = e_lo + me + 2k
        LeducHand h;
        bool live = false;
        int64_t e = -1;
        uint64_t g = 0;
        int t = 0;
        long long s1 = 0, s2 = 0, nd = 0;
        if (tid < kSlots) {
            e = e_lo + me + 2 * (int64_t)tid;
            live = e < e_hi;
            if (live) {
                g = (uint64_t)pair * (uint64_t)a.n_episodes + (uint64_t)e;
                leduc_deal(h, g, a.seed);
            }
        }
        if (tid == 0) next_k = kSlots;

        while (true) {
            // rank this CTA's live hands by acting seat
            const int seat = live ? h.actor : -1;
            const unsigned b0 = __ballot_sync(0xffffffffu, seat == 0);
            const unsigned b1 = __ballot_sync(0xffffffffu, seat == 1);
            if (lane == 0) { wcnt[0][warp] = __popc(b0); wcnt[1][warp] = __popc(b1); }
            __syncthreads();
            int pre = 0, c0 = 0, c1 = 0;
#pragma unroll
            for (int w = 0; w < 8; ++w) {
                c0 += wcnt[0][w];
                c1 += wcnt[1][w];
                if (w < warp) pre += seat == 1 ? wcnt[1][w] : wcnt[0][w];
            }
            const unsigned mine = seat == 1 ? b1 : b0;
            const int rank = pre + __popc(mine & ((1u << lane) - 1u));
            const bool placed = live && rank < kPart;
            float ob[17];
            float u = 0.f;
            // Every (target CTA, row) slot of this CTA's part of both tiles is
            // written each step: by its placed hand, else with zeros, so each
            // target receives a fixed byte count.
            if (placed) {
                u = u24(draw(g, (uint32_t)t, (uint32_t)seat, a.seed).x);   // ready before the logits
                leduc_obs(h, ob);
                uint32_t w[16];
#pragma unroll
                for (int i = 0; i < 8; ++i) w[i] = tc::pack_bf16(ob[2 * i], ob[2 * i + 1]);
                w[8] = tc::pack_bf16(ob[16], 0.f);
#pragma unroll
                for (int i = 9; i < 16; ++i) w[i] = 0u;
                const uint32_t bar = cl::map(&x_bar, (uint32_t)seat);
#pragma unroll
                for (int c = 0; c < 4; ++c)
                    cl::st_async_v4(cl::map(smem + Eng::kAct + Eng::act_offset((int)me * kPart + rank, 8 * c),
                                            (uint32_t)seat),
                                    make_uint4(w[4 * c], w[4 * c + 1], w[4 * c + 2], w[4 * c + 3]), bar);
            }
            if (tid < 2 * kPart) {
                const int tgt = tid / kPart, rk = tid % kPart;
                if (rk >= min(tgt == 0 ? c0 : c1, kPart)) {
                    const uint32_t bar = cl::map(&x_bar, (uint32_t)tgt);
#pragma unroll
                    for (int c = 0; c < 4; ++c)
                        cl::st_async_v4(cl::map(smem + Eng::kAct + Eng::act_offset((int)me * kPart + rk, 8 * c),
                                                (uint32_t)tgt),
                                        make_uint4(0, 0, 0, 0), bar);
                }
            }
            if (tid < 2) {                  // header to CTA tid: rows placed there, live hands here
                const uint32_t n = (uint32_t)min(tid == 0 ? c0 : c1, kPart);
                cl::st_async_v4(cl::map(&hdr[me], (uint32_t)tid), make_uint4(n, (uint32_t)(c0 + c1), 0, 0),
                                cl::map(&x_bar, (uint32_t)tid));
            }
            // Thread 0 waits (bounded) and decides for the CTA; the barrier
            // passes its view of the received data to every thread.
            if (tid == 0) {
                if (!dead_s && !cl::wait_cluster_bounded(&x_bar, x_par, kWaitLimitNs)) {
                    dead_s = 1u;
                    atomicOr(a.err, ERRBIT_TIMEOUT);
                }
                mbar_arrive_expect_tx(&x_bar, kXTx);                      // armed for the next step
                go_s = (!dead_s && (hdr[0].y != 0 || hdr[1].y != 0)) ? 1u : 0u;
            }
            x_par ^= 1u;
            __syncthreads();
            if (!go_s) break;
            // The tile rows arrived as generic-proxy stores; the MMA issuer
            // orders them before the tensor core's reads (forward's opening fence).
            Eng::forward(smem, nullptr, tbase, &mma_bar, mma_par, a.err, [&](int r, const float* lg) {
                const uint32_t src = (uint32_t)(r / kPart);
                cl::st_async_v4(cl::map(lgbuf + (me * kPart + r % kPart) * 4, src),
                                make_uint4(__float_as_uint(lg[0]), __float_as_uint(lg[1]),
                                           __float_as_uint(lg[2]), 0u),
                                cl::map(&lg_bar, src));
            }, /*x_published=*/true);
            if (tid == 0) {
                if (!dead_s && !cl::wait_cluster_bounded(&lg_bar, lg_par, kWaitLimitNs)) {
                    dead_s = 1u;
                    atomicOr(a.err, ERRBIT_TIMEOUT);
                }
                mbar_arrive_expect_tx(&lg_bar, kLgTx);
            }
            lg_par ^= 1u;
            __syncthreads();
            if (dead_s) break;
            if (placed) {
                const float* lp = lgbuf + (seat * kPart + rank) * 4;
                float lg[3] = {lp[0], lp[1], lp[2]};
                const unsigned legal = leduc_legal(h);
                const int act = sample_masked<3>(lg, legal, u);
                const bool rec = e < a.n_dump;
                const int64_t rb = ((int64_t)pair * a.n_dump + e) * kMaxDec;
                if (rec) {
                    if (a.d_obs) {
                        float* o = a.d_obs + (rb + t) * 20;
#pragma unroll
                        for (int i = 0; i < 17; ++i) o[i] = ob[i];
                        o[17] = 0.f; o[18] = 0.f; o[19] = 0.f;
                    }
                    if (a.d_logits) {
                        float* l = a.d_logits + (rb + t) * 3;
                        l[0] = lg[0]; l[1] = lg[1]; l[2] = lg[2];
                    }
                    if (a.d_action) a.d_action[rb + t] = (uint8_t)act;
                }
                leduc_apply(h, act);
                if (rec) {
                    if (a.d_reward) a.d_reward[rb + t] = h.done ? (float)h.payoff : 0.f;
                    if (a.d_done) a.d_done[rb + t] = h.done ? 1 : 0;
                }
                ++t;
                ++nd;
                if (h.done) {
                    s1 += h.payoff;
                    s2 += (long long)h.payoff * h.payoff;
                    if (rec) {
                        for (int k = t; k < kMaxDec; ++k) {
                            if (a.d_obs)
                                for (int i = 0; i < 20; ++i) a.d_obs[(rb + k) * 20 + i] = 0.f;
                            if (a.d_logits)
                                for (int i = 0; i < 3; ++i) a.d_logits[(rb + k) * 3 + i] = 0.f;
                            if (a.d_action) a.d_action[rb + k] = 255;
                            if (a.d_reward) a.d_reward[rb + k] = 0.f;
                            if (a.d_done) a.d_done[rb + k] = 1;
                        }
                    }
                    const int64_t k = (int64_t)atomicAdd(&next_k, 1ull);
                    e = e_lo + me + 2 * k;
                    live = e < e_hi;
                    if (live) {
                        g = (uint64_t)pair * (uint64_t)a.n_episodes + (uint64_t)e;
                        leduc_deal(h, g, a.seed);
                        t = 0;
                    }
                }
            }
            ++step;
        }
        block_add_sums(s1, s2, nd, a.acc + 2 * pair, a.n_dec);
        if (dead_s) break;          // uniform: written only before a barrier
    }
    tc::fence_before_sync();
    __syncthreads();
    cluster_barrier_all();          // no peer touches this CTA's shared memory after this
    if (warp == 0) tc::tmem_dealloc(tbase, Eng::kTmemCols);
}

}  // namespace

uint32_t leduc_tc_policy_floats() { return Eng::kPolicyBytes / 4; }

cudaError_t launch_leduc_eval_tc(const EvalArgs& a, int n_sm, cudaStream_t s) {
    if (a.n_pairs == 0) return cudaSuccess;
    cudaError_t err = cudaFuncSetAttribute(leduc_eval_tc_kernel,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmem);
    if (err != cudaSuccess) return err;
    const int64_t total = (int64_t)a.n_pairs * a.n_episodes;
    int64_t clusters = (total + 2 * kSlots - 1) / (2 * kSlots);
    const int64_t max_clusters = n_sm / 2;
    if (clusters > max_clusters) clusters = max_clusters;
    if (clusters < 1) clusters = 1;
    leduc_eval_tc_kernel<<<(unsigned)(2 * clusters), kThreads, kSmem, s>>>(a);
    return cudaGetLastError();
}

}  // namespace malib
