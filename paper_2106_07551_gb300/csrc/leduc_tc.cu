// Payoff-table evaluation of Leduc hold'em with bf16 MLP policies on the
// tensor cores (Sec. 3.2 payoff table, Sec. 4.2 Monte-Carlo simulations per
// policy combination).
//
// Work units are (pair, segment of at most kMaxHands hands), claimed by the
// CTAs from a counter. A CTA plays a unit's hands all at once, in phases: in a
// phase every live hand whose acting seat is s makes one decision, through
// seat s's policy, which is the only policy in shared memory; phases alternate
// between the seats (a phase without hands is skipped), and the policy is
// restaged between them. So every tile of the tensor-core forward holds 128
// decisions of one policy, and one policy at a time fits the shared memory
// with the pipelined engine's buffers.
// Hands live in global memory (a state word pair per hand, in the CTA's part
// of the context's work space); each seat has two queues of hand slots: the
// phase of seat s takes the current queue of s whole, hands that act next as
// the other seat join its current queue, hands that act again as s join the
// other queue of s, which becomes current when the phase ends (queues never
// change while they are read). The phase of a unit's first decisions deals the
// hands from their Philox keys.
// Warps, in warpgroups (setmaxnreg moves registers between them):
//  * the engine's two epilogue teams (mlp_tc2.cuh), then a warpgroup whose
//    first two warps hold its MMA threads (two idle);
//  * producers (4 warps): one row per thread, the hand's observation into a
//    bf16 tile (feature 15, constant 1, is folded into b1);
//  * consumers (4 warps): one row per thread, the logits (partials + b3), the
//    masked softmax draw keyed by (episode, decision, seat), the transition,
//    the payoff sums of finished hands, the queue of the next acting seat.
// Every wait is bounded.
#include "device_common.cuh"
#include "eval_common.cuh"
#include "internal.h"
#include "leduc_env.cuh"
#include "mlp_tc2.cuh"

namespace malib {

namespace {

constexpr int kK1 = 16;                    // observation inputs after folding feature 15
constexpr int kTW = 8;                     // epilogue warps per engine slot
using E = Eng2<kK1, 3, 3, kTW>;
constexpr int kEpiWG = kTW / 2;            // warpgroups of the two epilogue teams
constexpr int kMmaWG = kEpiWG, kProdWG = kEpiWG + 1, kConsWG = kEpiWG + 2;
constexpr int kWarps = 4 * (kEpiWG + 3);
constexpr int kThreads = 32 * kWarps;
constexpr int kProdWarp = 4 * kProdWG, kConsWarp = 4 * kConsWG;
// registers per thread after setmaxnreg: epilogue, MMA, producer, consumer
// warpgroups (their sum over the CTA stays within the launch's allocation)
constexpr int kRegEpi = kTW == 8 ? 80 : 112, kRegMma = kTW == 8 ? 48 : 56, kRegProd = kTW == 8 ? 48 : 64,
              kRegCons = kTW == 8 ? 88 : 128;
constexpr int kRegLaunch = 65536 / kThreads / 8 * 8;   // the launch's registers per thread
static_assert((kEpiWG * kRegEpi + kRegMma + kRegProd + kRegCons) <= (kEpiWG + 3) * kRegLaunch,
              "register split within the launch's allocation");

constexpr int kMaxDec = 8;
constexpr uint32_t kX = (E::kImage + 1023u) / 1024u * 1024u;     // X tiles
constexpr uint32_t kP = kX + E::kNX * E::kXBytes;                  // partial logits
constexpr uint32_t kSmem = kP + 2 * E::kPBytes;
static_assert(kSmem <= 227 * 1024, "fits one CTA's shared memory");

// A hand in global memory: cards, round, raises, actions this round, actor,
// decisions so far (x) and both contributions (y).
__device__ __forceinline__ uint2 pack(const LeducHand& h, int t) {
    uint2 w;
    w.x = (uint32_t)h.c0 | ((uint32_t)h.c1 << 4) | ((uint32_t)h.pub << 8) | ((uint32_t)h.round << 12) |
          ((uint32_t)h.raises << 13) | ((uint32_t)h.nact << 15) | ((uint32_t)h.actor << 17) |
          ((uint32_t)t << 18);
    w.y = (uint32_t)h.con0 | ((uint32_t)h.con1 << 8);
    return w;
}
__device__ __forceinline__ void unpack(uint2 w, LeducHand& h, int& t) {
    h.c0 = (int)(w.x & 15u);
    h.c1 = (int)((w.x >> 4) & 15u);
    h.pub = (int)((w.x >> 8) & 15u);
    h.round = (int)((w.x >> 12) & 1u);
    h.raises = (int)((w.x >> 13) & 3u);
    h.nact = (int)((w.x >> 15) & 3u);
    h.actor = (int)((w.x >> 17) & 1u);
    t = (int)((w.x >> 18) & 15u);
    h.con0 = (int)(w.y & 255u);
    h.con1 = (int)((w.y >> 8) & 255u);
    h.done = 0;
    h.payoff = 0;
}

struct Ctl {                   // per-CTA control words (shared memory)
    int64_t unit;              // claimed unit, or -1 when none is left
    int pair, p0, p1, ok;
    int64_t e_lo;              // first hand of the unit
    int n;                     // hands of the unit
    int cur[2];                // current queue of each seat (0 or 1)
    int len[2][2];             // [seat][queue] entries
    int seat;                  // seat of the current phase
    int first;                 // 1 in the unit's first phase (hands are dealt)
    int staged;                // policy id in shared memory (-1: none)
    uint32_t stagings;         // policies staged so far (stage barrier phase)
};

// What every role needs of the current phase.
struct Phase {
    int pair, s, n;
    int64_t e_lo;
    uint32_t tile;             // the phase's first tile (over the whole kernel)
    uint32_t nt;               // tiles of the phase
    bool first;                // hands are dealt in this phase
    const uint16_t* qin;       // queue read by the phase (not used when first)
};

// The unit and phase loop, run by every role in its own copy (each copy
// compiled within its warpgroup's register budget); all copies pass the same
// CTA barriers in the same order; wait_stage: the role waits for a new policy
// image to land before its phase. on_phase(ph) does the role's share of a
// phase, on_stage() its work after a new policy has landed, on_unit(sums)
// adds the unit's payoff sums (consumers hold them; the others add zeros).
template <class OnPhase, class OnStage>
__device__ __forceinline__ void drive(const EvalArgs& a, const LeducWork& w, E::Bars& bars, Ctl& ctl,
                                      uint8_t* smem, OnPhase&& on_phase, OnStage&& on_stage,
                                      long long* sums, bool wait_stage = true) {
    const int tid = threadIdx.x;
    const int64_t n_seg = w.n_seg;
    const int64_t n_units = w.n_units;
    const int64_t n_whole = (int64_t)w.split_from * n_seg;   // units before the split pairs
    uint16_t* q_base = w.queues + (size_t)blockIdx.x * 4 * w.max_hands;   // [seat][queue][max_hands]
    uint32_t tile = 0;
    while (true) {
        __syncthreads();                         // ctl of the previous unit is read by all
        if (tid == 0) {
            const int64_t u = (int64_t)atomicAdd(a.work, 1ull);
            ctl.unit = u < n_units ? u : -1;
            if (u < n_units) {
                // pairs before split_from in n_seg segments, the others in 2 n_seg
                const bool split = u >= n_whole;
                const int64_t ns = split ? 2 * n_seg : n_seg;
                const int64_t v = split ? u - n_whole : u;
                const int pair = (int)(split ? w.split_from + v / ns : v / ns);
                const int64_t seg = v % ns;
                const int64_t per = (a.n_episodes + ns - 1) / ns;
                ctl.pair = pair;
                ctl.e_lo = seg * per;
                const int64_t hi = min(a.n_episodes, ctl.e_lo + per);
                ctl.n = (int)max((int64_t)0, hi - ctl.e_lo);
                ctl.p0 = a.pairs[2 * pair];
                ctl.p1 = a.pairs[2 * pair + 1];
                ctl.ok = pair_ok(a, ctl.p0, ctl.p1) ? 1 : 0;
                if (!ctl.ok && seg == 0) atomicOr(a.err, ERRBIT_BAD_PAIR);
                ctl.cur[0] = ctl.cur[1] = 0;
                ctl.len[0][0] = ctl.n;          // seat 0 acts first in every hand
                ctl.len[0][1] = ctl.len[1][0] = ctl.len[1][1] = 0;
                ctl.seat = 0;
                ctl.first = 1;
            }
        }
        __syncthreads();
        if (ctl.unit < 0) break;
        if (!ctl.ok || ctl.n == 0) continue;
        sums[0] = sums[1] = sums[2] = 0;
        while (true) {
            const int s = ctl.seat;
            const int n = ctl.len[s][ctl.cur[s]];
            if (n == 0 && ctl.len[s ^ 1][ctl.cur[s ^ 1]] == 0) break;   // the unit is done
            const int pol = s == 0 ? ctl.p0 : ctl.p1;
            const bool restage = n > 0 && pol != ctl.staged;
            if (restage) {
                // every MMA and epilogue read of the previous policy is done (the
                // previous phase ended with a CTA barrier); ctl is written again
                // only after the next CTA barrier
                if (tid == 0) E::stage(smem, reinterpret_cast<const uint8_t*>(a.arena + a.pol_offset[pol]), bars);
                // the producers and consumers do not wait: the producers' tiles do
                // not depend on the policy (they build the phase's first tiles while
                // it lands), and the consumers read the image (b3) only after a
                // p_full, which the engine announces after it has waited for it
                if (wait_stage) E::wait(bars, &bars.stage, ctl.stagings & 1u, a.err);
                on_stage();
            }
            if (n > 0) {
                Phase ph;
                ph.pair = ctl.pair;
                ph.s = s;
                ph.n = n;
                ph.e_lo = ctl.e_lo;
                ph.tile = tile;
                ph.nt = (uint32_t)((n + 127) / 128);
                ph.first = ctl.first != 0;
                ph.qin = q_base + (size_t)(2 * s + ctl.cur[s]) * w.max_hands;
                on_phase(ph);
                tile += ph.nt;
            }
            __syncthreads();                     // every role has finished the phase
            if (tid == 0) {
                if (restage) {
                    ctl.staged = pol;
                    ++ctl.stagings;
                }
                if (n > 0) {
                    ctl.len[s][ctl.cur[s]] = 0;  // the queue just read is empty
                    ctl.cur[s] ^= 1;             // hands that act again as s
                    ctl.first = 0;
                }
                ctl.seat = s ^ 1;
            }
            __syncthreads();
            if (E::is_dead(bars)) break;
        }
        block_add_sums(sums[0], sums[1], sums[2], a.acc + 2 * ctl.pair, a.n_dec);
        if (E::is_dead(bars)) break;
    }
}

// The CTA's last barrier (every MMA has completed: the MMA threads waited for
// their last commits), then warp 0 releases the tensor memory. Called at the
// end of every role's branch, inside its register budget.
__device__ __forceinline__ void end_cta(uint32_t tbase) {
    tc::fence_before_sync();
    __syncthreads();
    if ((threadIdx.x >> 5) == 0) tc::tmem_dealloc(tbase, E::kTmemCols);
}

// kDump: the call records its first n_dump hands of every pair (the consumers'
// recording code is compiled out of the other instance).
template <bool kDump>
__global__ void __launch_bounds__(kThreads, 1) leduc_eval_tc_kernel(EvalArgs a, LeducWork w) {
    extern __shared__ __align__(1024) uint8_t smem[];
    __shared__ E::Bars bars;
    __shared__ Ctl ctl;
    __shared__ uint32_t tmem_base;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int wg = warp >> 2;

    if (tid == 0) {
        bars.init();
        ctl.staged = -1;
        ctl.stagings = 0;
    }
    if (warp == 0) {
        tc::tmem_alloc(&tmem_base, E::kTmemCols);
        tc::tmem_relinquish();
    }
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    const uint32_t tbase = tmem_base;
    long long sums[3] = {0, 0, 0};
    auto nothing = [] {};

    if (wg < kEpiWG) {
        // ---- epilogue teams (warps 0 .. kTW - 1 slot 0, then slot 1)
        tc::set_max_regs<kRegEpi, kRegLaunch>();
        if (warp < kTW) {
            E::Epilogue<0> ep;
            ep.p_base_off = kP;
            drive(a, w, bars, ctl, smem, [&](const Phase& ph) { ep.run(smem, tbase, bars, ph.nt, a.err); },
                  [&] { ep.init(smem); }, sums);
        } else {
            E::Epilogue<1> ep;
            ep.p_base_off = kP;
            drive(a, w, bars, ctl, smem, [&](const Phase& ph) { ep.run(smem, tbase, bars, ph.nt, a.err); },
                  [&] { ep.init(smem); }, sums);
        }
        end_cta(tbase);
    } else if (wg == kMmaWG) {
        // ---- the MMA threads (the warpgroup's first two warps; two idle)
        tc::set_max_regs<kRegMma, kRegLaunch>();
        if (warp == 4 * kMmaWG) {
            E::Issuer<0> is;
            drive(a, w, bars, ctl, smem, [&](const Phase& ph) {
                if (lane == 0) is.run(smem, smem_u32(smem + kX), tbase, bars, ph.nt, a.err);
            }, nothing, sums);
            if (lane == 0) is.finish(bars, a.err);
        } else if (warp == 4 * kMmaWG + 1) {
            E::Issuer<1> is;
            drive(a, w, bars, ctl, smem, [&](const Phase& ph) {
                if (lane == 0) is.run(smem, smem_u32(smem + kX), tbase, bars, ph.nt, a.err);
            }, nothing, sums);
            if (lane == 0) is.finish(bars, a.err);
        } else {
            drive(a, w, bars, ctl, smem, [](const Phase&) {}, nothing, sums);
        }
        end_cta(tbase);
    } else if (wg == kProdWG) {
        // ---- producers: observation rows, one per thread
        tc::set_max_regs<kRegProd, kRegLaunch>();
        const int r = tid - kProdWarp * 32;
        const uint2* hands = w.hands + (size_t)blockIdx.x * w.max_hands;
        drive(a, w, bars, ctl, smem, [&](const Phase& ph) {
            // the next tile's hand (queue entry, state) is loaded before this
            // tile's wait, so that its global-memory latency overlaps
            int nslot = r;
            uint2 nst = make_uint2(0, 0);
            if (!ph.first && r < ph.n) {
                nslot = (int)ph.qin[r];
                nst = hands[nslot];
            }
            for (uint32_t i = 0; i < ph.nt; ++i) {
                const uint32_t T = ph.tile + i;
                const int buf = (int)(T % E::kNX);
                const int idx = (int)i * 128 + r;
                const int slot = nslot;
                const uint2 st = nst;
                const int nidx = idx + 128;
                if (nidx < ph.n) {
                    nslot = ph.first ? nidx : (int)ph.qin[nidx];
                    if (!ph.first) nst = hands[nslot];
                }
                uint32_t wv[8] = {0, 0, 0, 0, 0, 0, 0, 0};
                if (idx < ph.n) {
                    LeducHand h;
                    int t;
                    if (ph.first) {
                        leduc_deal(h, (uint64_t)ph.pair * (uint64_t)a.n_episodes + (uint64_t)(ph.e_lo + slot), a.seed);
                        t = 0;
                    } else {
                        unpack(st, h, t);
                    }
                    float ob[17];
                    leduc_obs(h, ob);
#pragma unroll
                    for (int q = 0; q < 7; ++q) wv[q] = tc::pack_bf16(ob[2 * q], ob[2 * q + 1]);
                    wv[7] = tc::pack_bf16(ob[14], ob[16]);   // feature 15 is folded into b1
                }
                if (T >= (uint32_t)E::kNX) E::wait(bars, &bars.x_free[buf], ((T / E::kNX) - 1) & 1u, a.err);
                uint8_t* xt = smem + kX + buf * E::kXBytes;
                *reinterpret_cast<uint4*>(xt + E::x_offset(r, 0)) = make_uint4(wv[0], wv[1], wv[2], wv[3]);
                *reinterpret_cast<uint4*>(xt + E::x_offset(r, 8)) = make_uint4(wv[4], wv[5], wv[6], wv[7]);
                fence_proxy_async_smem();
                asm volatile("bar.sync 2, 128;" ::: "memory");
                if (r == 0) mbar_arrive_release(&bars.x_full[buf]);
            }
        }, nothing, sums, /*wait_stage=*/false);
        end_cta(tbase);
    } else {
        // ---- consumers: draw, transition, sums, next queue; one row per thread
        tc::set_max_regs<kRegCons, kRegLaunch>();
        const int r = tid - kConsWarp * 32;
        uint2* hands = w.hands + (size_t)blockIdx.x * w.max_hands;
        uint16_t* q_base = w.queues + (size_t)blockIdx.x * 4 * w.max_hands;
        drive(a, w, bars, ctl, smem, [&](const Phase& ph) {
            const float* b3 = reinterpret_cast<const float*>(smem + E::kB3);
            const int s = ph.s;
            // the next tile's hand is loaded before this tile's wait
            int nslot = r;
            uint2 nst = make_uint2(0, 0);
            if (!ph.first && r < ph.n) {
                nslot = (int)ph.qin[r];
                nst = hands[nslot];
            }
            for (uint32_t i = 0; i < ph.nt; ++i) {
                const uint32_t T = ph.tile + i;
                const int sl = (int)(T & 1u);
                const int cslot = nslot;
                const uint2 cst = nst;
                {
                    const int nidx = (int)i * 128 + 128 + r;
                    if (nidx < ph.n) {
                        nslot = ph.first ? nidx : (int)ph.qin[nidx];
                        if (!ph.first) nst = hands[nslot];
                    }
                }
                E::wait(bars, &bars.p_full[sl], (T >> 1) & 1u, a.err);
                const float* pp = reinterpret_cast<const float*>(smem + kP + sl * E::kPBytes);
                const int idx = (int)i * 128 + r;
                float lg[3] = {0.f, 0.f, 0.f};
                if (idx < ph.n) {
#pragma unroll
                    for (int q = 0; q < 3; ++q)
                        lg[q] = __fadd_rn(E::kSplit == 2 ? __fadd_rn(pp[r * 3 + q], pp[(128 + r) * 3 + q])
                                                          : pp[r * 3 + q],
                                          b3[q]);
                }
                asm volatile("bar.sync 3, 128;" ::: "memory");
                if (r == 0) mbar_arrive_release(&bars.p_free[sl]);
                int next = -1, slot = 0;
                if (idx < ph.n) {
                    slot = cslot;
                    LeducHand h;
                    int t;
                    const int64_t e = ph.e_lo + slot;
                    const uint64_t gid = (uint64_t)ph.pair * (uint64_t)a.n_episodes + (uint64_t)e;
                    if (ph.first) {
                        leduc_deal(h, gid, a.seed);
                        t = 0;
                    } else {
                        unpack(cst, h, t);
                    }
                    const float u = u24(draw(gid, (uint32_t)t, (uint32_t)s, a.seed).x);
                    const unsigned legal = leduc_legal(h);
                    const int act = sample_masked<3>(lg, legal, u);
                    const bool rec = kDump && e < a.n_dump;
                    const int64_t rb = ((int64_t)ph.pair * a.n_dump + e) * kMaxDec;
                    if (rec) {
                        if (a.d_obs) {
                            float ob[17];
                            leduc_obs(h, ob);
                            float* o = a.d_obs + (rb + t) * 20;
#pragma unroll
                            for (int q = 0; q < 17; ++q) o[q] = ob[q];
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
                    ++sums[2];
                    if (h.done) {
                        sums[0] += h.payoff;
                        sums[1] += (long long)h.payoff * h.payoff;
                        if (rec) {
                            for (int k = t; k < kMaxDec; ++k) {
                                if (a.d_obs)
                                    for (int q = 0; q < 20; ++q) a.d_obs[(rb + k) * 20 + q] = 0.f;
                                if (a.d_logits)
                                    for (int q = 0; q < 3; ++q) a.d_logits[(rb + k) * 3 + q] = 0.f;
                                if (a.d_action) a.d_action[rb + k] = 255;
                                if (a.d_reward) a.d_reward[rb + k] = 0.f;
                                if (a.d_done) a.d_done[rb + k] = 1;
                            }
                        }
                    } else {
                        hands[slot] = pack(h, t);
                        next = h.actor;
                    }
                }
                // the hand joins the queue of its next acting seat: the other
                // seat's current queue, or this seat's other queue
#pragma unroll
                for (int ns = 0; ns < 2; ++ns) {
                    const unsigned m = __ballot_sync(0xffffffffu, next == ns);
                    if (m == 0u) continue;
                    const int qi = ns == s ? (ctl.cur[s] ^ 1) : ctl.cur[ns];
                    const int leader = __ffs(m) - 1;
                    int base = 0;
                    if (lane == leader) base = atomicAdd(&ctl.len[ns][qi], __popc(m));
                    base = __shfl_sync(0xffffffffu, base, leader);
                    if (next == ns)
                        q_base[(size_t)(2 * ns + qi) * w.max_hands + base + __popc(m & ((1u << lane) - 1u))] =
                            (uint16_t)slot;
                }
            }
        }, nothing, sums, /*wait_stage=*/false);
        end_cta(tbase);
    }
}

}  // namespace

int64_t leduc_tc_units(int32_t n_pairs, int64_t n_episodes, int n_sm, int64_t* n_seg_out,
                       int32_t* split_from_out) {
    int64_t n_seg = (n_episodes + kLeducTcMaxHands - 1) / kLeducTcMaxHands;
    // enough units for every SM when pairs are few
    while ((int64_t)n_pairs * n_seg < n_sm && (n_episodes + n_seg - 1) / n_seg > 256) ++n_seg;
    // when there are more pairs than SMs, the last n_sm pairs (the last units
    // claimed) are played in halves: a unit's time varies with its policies,
    // and shorter last units leave the CTAs closer together at the end
    int32_t split_from = n_pairs;
    if ((int64_t)n_pairs > n_sm && (n_episodes + 2 * n_seg - 1) / (2 * n_seg) >= 256) split_from = n_pairs - n_sm;
    *n_seg_out = n_seg;
    *split_from_out = split_from;
    return (int64_t)split_from * n_seg + (int64_t)(n_pairs - split_from) * 2 * n_seg;
}

cudaError_t launch_leduc_eval_tc(const EvalArgs& a, const LeducWork& w, int n_sm, cudaStream_t s) {
    if (a.n_pairs == 0) return cudaSuccess;
    auto kern = a.n_dump > 0 ? leduc_eval_tc_kernel<true> : leduc_eval_tc_kernel<false>;
    cudaError_t err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmem);
    if (err != cudaSuccess) return err;
    int64_t n_seg = 0;
    int32_t split_from = 0;
    const int64_t units = leduc_tc_units(a.n_pairs, a.n_episodes, n_sm, &n_seg, &split_from);
    const int64_t grid = units < n_sm ? units : n_sm;
    LeducWork ww = w;
    ww.n_seg = n_seg;
    ww.split_from = split_from;
    ww.n_units = units;
    kern<<<(unsigned)grid, kThreads, kSmem, s>>>(a, ww);
    return cudaGetLastError();
}

}  // namespace malib
