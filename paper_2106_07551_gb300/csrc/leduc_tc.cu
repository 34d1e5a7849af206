// Payoff-table evaluation of Leduc hold'em with bf16 MLP policies on the
// tensor cores (Sec. 3.2 payoff table, Sec. 4.2 Monte-Carlo simulations per
// policy combination).
//
// A cluster of two CTAs evaluates one pair at a time. CTA r keeps the policy of
// seat r resident in shared memory (bf16 weight image and biases, ~146 KB);
// the MLP's hidden activations stay in tensor memory.
// Each CTA has 16 warps in three roles:
//  * warps 0-7, the engine: runs 128-row tiles through the tensor-core MLP,
//    alternating between two hand groups, and returns every row's logits;
//  * warps 8-11 and 12-15, hand groups 0 and 1, 128 hands each. While the
//    engine works on one group's tile, the other group samples its actions,
//    applies them, deals new hands and publishes its next observations, so the
//    environment work overlaps the tensor-core forward.
// Rows 64 s .. 64 s + 63 of a group's tile in CTA r hold observations of CTA s's
// hands acting as seat r, ranked with warp ballots (a hand beyond 64 waits a
// step; its randomness depends only on its own ids, so deferral changes no
// result). Observations (with a 16-byte header: rows placed, live hands) and
// logits travel as asynchronous stores into the peer's shared memory that
// complete transaction bytes on the receiver's mbarrier; every slot is written
// every step (unused rows with zeros), so each receiver expects a fixed byte
// count. A logits message whose flag is set tells a group that its hands of the
// segment are finished in both CTAs. Both CTAs walk the same pair segments
// (cluster c takes every n_cl-th pair); the engine restages weights when both
// groups have finished a segment.
// Control decisions of a role are taken by one thread and handed to the role
// through its own barrier, so every thread of a role takes the same path.
#include "cluster.cuh"
#include "device_common.cuh"
#include "eval_common.cuh"
#include "internal.h"
#include "leduc_env.cuh"
#include "mlp_tc.cuh"

namespace malib {

namespace {

constexpr int kK1 = 16;                    // observation inputs after folding feature 15
using Eng = MlpTc<kK1, 256, 16, true, /*kBarId=*/1>;
constexpr int kThreads = 512;
constexpr int kEngineThreads = 256;
constexpr int kGroups = 2;
constexpr int kSlots = 128;               // hands per group per CTA
constexpr int kPart = 64;                 // tile rows per source CTA
constexpr uint32_t kXBytes = Eng::kXBytes;                // one group's observation tile
constexpr uint32_t kX = Eng::kSmemBytes;                  // X tiles [group]
constexpr uint32_t kLg = kX + kGroups * kXBytes;          // logits [group][target][rank][4] fp32
constexpr uint32_t kSmem = kLg + kGroups * 2 * kPart * 16;
constexpr uint32_t kXTx = 2 * (kPart * kK1 * 2 + 16);     // rows + headers received per step
constexpr uint32_t kLgTx = 2 * kPart * 16;                // logits received per step
constexpr uint32_t kDoneFlag = 0x3f800000u;               // 1.0f in a logits row's 4th word
constexpr int kMaxDec = 8;
static_assert(kX % 16 == 0 && kLg % 16 == 0, "16-byte aligned tiles");

__device__ __forceinline__ void cluster_barrier_all() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n"
                 "barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

__device__ __forceinline__ void group_sync(int g) {
    if (g == 0) asm volatile("bar.sync 2, 128;" ::: "memory");
    else asm volatile("bar.sync 3, 128;" ::: "memory");
}

__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
    leduc_eval_tc_kernel(EvalArgs a) {
    extern __shared__ __align__(128) uint8_t smem[];
    __shared__ __align__(8) uint64_t stage_bar;
    __shared__ __align__(8) uint64_t mma_bar[2];
    __shared__ __align__(8) uint64_t x_bar[kGroups];    // a group's rows and headers
    __shared__ __align__(8) uint64_t lg_bar[kGroups];   // a group's logits
    __shared__ __align__(8) uint64_t h1_bar[kGroups][2];  // h1 of a group's tile stored ([0] used)
    __shared__ __align__(16) uint4 hdr[kGroups][2];     // [group][source CTA]: {rows here, live}
    __shared__ uint32_t tmem_base;
    __shared__ uint32_t dead_s;                         // a bounded wait expired
    __shared__ uint32_t eng_flag[2];                    // engine: 0 run, 1 group done, 2 stop
                                                        // (two slots, used alternately)
    __shared__ uint32_t grp_flag[kGroups];              // group: 0 logits, 1 segment done, 2 stop
    __shared__ int wcnt[kGroups][2][4];                 // [group][seat][warp of the group]
    __shared__ unsigned long long next_k[kGroups];
    __shared__ long long red[kGroups][3][4];

    float* lgbuf = reinterpret_cast<float*>(smem + kLg);
    const uint32_t me = cl::rank();
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

    if (tid == 0) {
        dead_s = 0u;
        mbar_init(&stage_bar, 1);
        mbar_init(&mma_bar[0], 1);
        mbar_init(&mma_bar[1], 1);
        for (int g = 0; g < kGroups; ++g) {
            mbar_init(&x_bar[g], 1);
            mbar_init(&lg_bar[g], 1);
            mbar_init(&h1_bar[g][0], 1);
            mbar_init(&h1_bar[g][1], 1);
            mbar_arrive_expect_tx(&x_bar[g], kXTx);         // armed for the first step
            mbar_arrive_expect_tx(&lg_bar[g], kLgTx);
        }
    }
    if (warp == 0) {
        tc::tmem_alloc(&tmem_base, Eng::kTmemCols);
        tc::tmem_relinquish();
    }
    for (uint32_t i = tid * 16; i < kGroups * kXBytes; i += kThreads * 16)
        *reinterpret_cast<uint4*>(smem + kX + i) = make_uint4(0, 0, 0, 0);
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    cluster_barrier_all();          // peers' barriers exist before any remote store
    const uint32_t tbase = tmem_base;

    // Work units: a pair's hands, cut into `parts` pieces when there are fewer
    // pairs than clusters. Cluster c takes units c, c + n_cl, ...: strided, so
    // that its pairs come from every row and column of the table (neighbouring
    // pairs share a policy and so have similar game lengths; contiguous ranges
    // left clusters with 10 % more work than others).
    const int64_t n_cl = gridDim.x / 2, cid = blockIdx.x / 2;
    const int64_t parts = a.n_pairs >= n_cl ? 1 : (n_cl + a.n_pairs - 1) / a.n_pairs;
    const int64_t chunk = (a.n_episodes + parts - 1) / parts;
    const int64_t n_units = (int64_t)a.n_pairs * parts;

    if (warp < 8) {
        // ------------------------------------------------------------ engine
        uint32_t stage_par = 0, mma_par = 0, x_bits = 0;      // x_bar parity of group g: bit g
        bool stop = false;
        for (int64_t u = cid; u < n_units && !stop; u += n_cl) {
            const int pair = (int)(u % a.n_pairs);
            const int64_t e_lo = (u / a.n_pairs) * chunk;
            const int64_t e_hi = min(a.n_episodes, e_lo + chunk);
            if (e_lo >= e_hi) continue;                     // the hand groups skip it too
            const int p0 = a.pairs[2 * pair], p1 = a.pairs[2 * pair + 1];
            if (!pair_ok(a, p0, p1)) continue;             // the hand groups skip it too
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
            tc::fence_before_sync();
            Eng::sync();
            uint32_t done_bits = 0, fslot = 0;
            while (done_bits != 3u && !stop) {
                for (int g = 0; g < kGroups && !stop; ++g) {
                    if (done_bits & (1u << g)) continue;
                    if (tid == 0) {
                        if (!dead_s && !cl::wait_cluster_bounded(&x_bar[g], (x_bits >> g) & 1u,
                                                                 kWaitLimitNs)) {
                            dead_s = 1u;
                            atomicOr(a.err, ERRBIT_TIMEOUT);
                        }
                        mbar_arrive_expect_tx(&x_bar[g], kXTx);   // armed for the group's next step
                        eng_flag[fslot] = dead_s ? 2u : ((hdr[g][0].y | hdr[g][1].y) == 0 ? 1u : 0u);
                    }
                    x_bits ^= 1u << g;
                    Eng::sync();
                    // a slot is rewritten two decisions later, after the next one's
                    // barrier, which every thread passes only once it has read it
                    const uint32_t f = eng_flag[fslot];
                    fslot ^= 1u;
                    if (f == 2u) { stop = true; break; }
                    if (f == 1u) {
                        // no live hand of the group in either CTA: tell both sources
                        done_bits |= 1u << g;
                        if (tid < 128) {
                            const uint32_t src = (uint32_t)(tid / kPart);
                            float* dst = lgbuf + ((g * 2 + (int)me) * kPart + tid % kPart) * 4;
                            cl::st_async_v4(cl::map(dst, src), make_uint4(0, 0, 0, kDoneFlag),
                                            cl::map(&lg_bar[g], src));
                        }
                        continue;
                    }
                    Eng::forward(smem, nullptr, tbase, mma_bar, mma_par, a.err,
                                 [&](int r, const float* lg) {
                                     const uint32_t src = (uint32_t)(r / kPart);
                                     float* dst = lgbuf + ((g * 2 + (int)me) * kPart + r % kPart) * 4;
                                     cl::st_async_v4(cl::map(dst, src),
                                                     make_uint4(__float_as_uint(lg[0]),
                                                                __float_as_uint(lg[1]),
                                                                __float_as_uint(lg[2]), 0u),
                                                     cl::map(&lg_bar[g], src));
                                 },
                                 smem_u32(smem + kX + g * kXBytes), /*x_published=*/true, h1_bar[g]);
                }
            }
        }
    } else {
        // ------------------------------------------------------------ hand groups
        const int g = (warp - 8) >> 2;                 // 0 or 1
        const int lt = tid - kEngineThreads - g * kSlots;
        const int gw = (warp - 8) & 3;                  // warp within the group
        uint32_t lg_par = 0, h1_par = 0;
        uint8_t* xg = smem + kX + g * kXBytes;
        bool stop = false;
        for (int64_t u = cid; u < n_units && !stop; u += n_cl) {
            const int pair = (int)(u % a.n_pairs);
            const int64_t e_lo = (u / a.n_pairs) * chunk;
            const int64_t e_hi = min(a.n_episodes, e_lo + chunk);
            if (e_lo >= e_hi) continue;                 // same decision in every role of both CTAs
            const int p0 = a.pairs[2 * pair], p1 = a.pairs[2 * pair + 1];
            if (!pair_ok(a, p0, p1)) {                  // same decision in every role of both CTAs
                if (tid == kEngineThreads && me == 0) atomicOr(a.err, ERRBIT_BAD_PAIR);
                continue;
            }
            // this group's hands: e = e_lo + me + 2 g + 4 k
            LeducHand h;
            int64_t e = e_lo + me + 2 * g + 4 * (int64_t)lt;
            bool live = e < e_hi;
            uint64_t gid = 0;
            int t = 0;
            long long s1 = 0, s2 = 0, nd = 0;
            if (live) {
                gid = (uint64_t)pair * (uint64_t)a.n_episodes + (uint64_t)e;
                leduc_deal(h, gid, a.seed);
            }
            if (lt == 0) next_k[g] = kSlots;
            while (true) {
                // rank this group's live hands by acting seat
                const int seat = live ? h.actor : -1;
                const unsigned b0 = __ballot_sync(0xffffffffu, seat == 0);
                const unsigned b1 = __ballot_sync(0xffffffffu, seat == 1);
                if (lane == 0) { wcnt[g][0][gw] = __popc(b0); wcnt[g][1][gw] = __popc(b1); }
                group_sync(g);
                int pre = 0, c0 = 0, c1 = 0;
#pragma unroll
                for (int w = 0; w < 4; ++w) {
                    c0 += wcnt[g][0][w];
                    c1 += wcnt[g][1][w];
                    if (w < gw) pre += seat == 1 ? wcnt[g][1][w] : wcnt[g][0][w];
                }
                const unsigned mine = seat == 1 ? b1 : b0;
                const int rank = pre + __popc(mine & ((1u << lane) - 1u));
                const bool placed = live && rank < kPart;
                float ob[17];
                float u = 0.f;
                if (placed) {
                    leduc_obs(h, ob);
                    uint32_t w[8];
#pragma unroll
                    for (int i = 0; i < 7; ++i) w[i] = tc::pack_bf16(ob[2 * i], ob[2 * i + 1]);
                    w[7] = tc::pack_bf16(ob[14], ob[16]);   // feature 15 is folded into b1
                    const uint32_t bar = cl::map(&x_bar[g], (uint32_t)seat);
#pragma unroll
                    for (int c = 0; c < 2; ++c)
                        cl::st_async_v4(cl::map(xg + Eng::x_offset((int)me * kPart + rank, 8 * c),
                                                (uint32_t)seat),
                                        make_uint4(w[4 * c], w[4 * c + 1], w[4 * c + 2], w[4 * c + 3]),
                                        bar);
                }
                {   // every unused slot of this CTA's part of both tiles gets zeros
                    const int tgt = lt / kPart, rk = lt % kPart;
                    if (rk >= min(tgt == 0 ? c0 : c1, kPart)) {
                        const uint32_t bar = cl::map(&x_bar[g], (uint32_t)tgt);
#pragma unroll
                        for (int c = 0; c < 2; ++c)
                            cl::st_async_v4(cl::map(xg + Eng::x_offset((int)me * kPart + rk, 8 * c),
                                                    (uint32_t)tgt),
                                            make_uint4(0, 0, 0, 0), bar);
                    }
                }
                if (lt < 2) {                                   // header to CTA lt
                    const uint32_t n = (uint32_t)min(lt == 0 ? c0 : c1, kPart);
                    cl::st_async_v4(cl::map(&hdr[g][me], (uint32_t)lt),
                                    make_uint4(n, (uint32_t)(c0 + c1), 0, 0),
                                    cl::map(&x_bar[g], (uint32_t)lt));
                }
                // the decision's uniform, drawn while the engines work
                if (placed) u = u24(draw(gid, (uint32_t)t, (uint32_t)seat, a.seed).x);
                // logits (or the end of the segment) from both engines. While
                // it waits, this group's leader issues the second output half of
                // layer 2 of the group's tile in this CTA once the engine has h1
                // in tensor memory (the engine's own MMA thread is then free for
                // its epilogue share); a forward needs it before it can finish.
                // (Issuing all of layer 2 from here measured 52.4 ms against
                // 49.4: the helper's response then delays layer 2's start.)
                if (lt == 0) {
                    bool pend = true;
                    const uint64_t t0 = globaltimer_ns();
                    while (!dead_s) {
                        if (pend && mbar_try_wait(&h1_bar[g][0], h1_par)) {
                            h1_par ^= 1u;
                            pend = false;
                            tc::fence_after_sync();
                            Eng::issue_layer2b(smem, tbase, &mma_bar[0]);
                        }
                        if (cl::try_wait_cluster(&lg_bar[g], lg_par)) break;
                        if (globaltimer_ns() - t0 > kWaitLimitNs) {
                            dead_s = 1u;
                            atomicOr(a.err, ERRBIT_TIMEOUT);
                        }
                    }
                    mbar_arrive_expect_tx(&lg_bar[g], kLgTx);
                    grp_flag[g] = dead_s ? 2u
                                         : (__float_as_uint(lgbuf[(g * 2) * kPart * 4 + 3]) == kDoneFlag
                                                ? 1u : 0u);
                }
                lg_par ^= 1u;
                group_sync(g);
                const uint32_t f = grp_flag[g];
                if (f != 0u) { stop = f == 2u; break; }
                if (placed) {
                    const float* lp = lgbuf + ((g * 2 + seat) * kPart + rank) * 4;
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
                    }
                }
                // finished hands take the group's next hands: one atomic per
                // warp, ranks within the warp from a ballot
                const bool need = placed && h.done;
                const unsigned nm = __ballot_sync(0xffffffffu, need);
                if (nm != 0u) {
                    const int leader = __ffs(nm) - 1;
                    unsigned long long base = 0ull;
                    if (lane == leader) base = atomicAdd(&next_k[g], (unsigned long long)__popc(nm));
                    base = __shfl_sync(0xffffffffu, base, leader);
                    if (need) {
                        const int64_t k = (int64_t)(base + (unsigned long long)__popc(nm & ((1u << lane) - 1u)));
                        e = e_lo + me + 2 * g + 4 * k;
                        live = e < e_hi;
                        if (live) {
                            gid = (uint64_t)pair * (uint64_t)a.n_episodes + (uint64_t)e;
                            leduc_deal(h, gid, a.seed);
                            t = 0;
                        }
                    }
                }
            }
            // the group's payoff sums: warp shuffles, then one atomic per sum
            s1 = warp_sum_ll(s1);
            s2 = warp_sum_ll(s2);
            nd = warp_sum_ll(nd);
            if (lane == 0) { red[g][0][gw] = s1; red[g][1][gw] = s2; red[g][2][gw] = nd; }
            group_sync(g);
            if (lt == 0) {
                long long t1 = 0, t2 = 0, t3 = 0;
                for (int w = 0; w < 4; ++w) { t1 += red[g][0][w]; t2 += red[g][1][w]; t3 += red[g][2][w]; }
                atomicAdd(a.acc + 2 * pair, (unsigned long long)t1);
                atomicAdd(a.acc + 2 * pair + 1, (unsigned long long)t2);
                atomicAdd(a.n_dec, (unsigned long long)t3);
            }
            group_sync(g);
        }
    }
    tc::fence_before_sync();
    __syncthreads();
    cluster_barrier_all();          // no peer touches this CTA's shared memory after this
    if (warp == 0) tc::tmem_dealloc(tbase, Eng::kTmemCols);
}

}  // namespace

cudaError_t launch_leduc_eval_tc(const EvalArgs& a, int n_sm, cudaStream_t s) {
    if (a.n_pairs == 0) return cudaSuccess;
    cudaError_t err = cudaFuncSetAttribute(leduc_eval_tc_kernel,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmem);
    if (err != cudaSuccess) return err;
    const int64_t total = (int64_t)a.n_pairs * a.n_episodes;
    int64_t clusters = (total + 2 * kGroups * kSlots - 1) / (2 * kGroups * kSlots);
    const int64_t max_clusters = n_sm / 2;
    if (clusters > max_clusters) clusters = max_clusters;
    if (clusters < 1) clusters = 1;
    leduc_eval_tc_kernel<<<(unsigned)(2 * clusters), kThreads, kSmem, s>>>(a);
    return cudaGetLastError();
}

}  // namespace malib
