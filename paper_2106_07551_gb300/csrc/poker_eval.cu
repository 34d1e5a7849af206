// Payoff-table evaluation for the poker games (Sec. 3.2 Evaluator, Sec. 4.2:
// each entry of the empirical payoff table is the Monte-Carlo mean over
// simulated hands of one policy combination).
//
// Kuhn: one thread per hand, tabular policies in registers.
// Leduc (fp32 MLP policies): a persistent CTA owns a contiguous range of
// (pair, hand) indices; both policies of the current pair are staged once into
// shared memory by bulk copy; 248 hand slots advance one decision per step; the
// observations of the slots are compacted by acting seat so every 4-row group
// of the MLP engine uses one policy; finished hands are replaced from the
// range at once so the slots stay full.
#include "device_common.cuh"
#include "internal.h"
#include "eval_common.cuh"
#include "leduc_env.cuh"
#include "mlp_f32.cuh"

namespace malib {

namespace {

// ---------------------------------------------------------------- Kuhn
// Cards J=0 < Q=1 < K=2, ante 1, one bet of 1. Infoset index card*2 + h with
// h = 1 when the seat faces a bet. Decision t uses counter (g, t, seat).
struct KuhnHand { int n; int act[3]; float p[3]; int payoff; };

// Entry idx of a 6-entry register table without dynamic indexing.
__device__ __forceinline__ float tab6(const float (&t)[6], int idx) {
    float v = t[0];
#pragma unroll
    for (int i = 1; i < 6; ++i) v = idx == i ? t[i] : v;
    return v;
}

// Seat 0 acts at decisions 0 and 2, seat 1 at decision 1, whatever the
// actions, so the three decision draws (g, t, seat) are known before the hand
// is played: they are drawn up front and the hand is resolved with selects, so
// the threads of a warp never run the generator on divergent paths. The third
// draw is used only after pass-bet.
__device__ __forceinline__ KuhnHand kuhn_play(const float (&t0)[6], const float (&t1)[6], uint64_t g,
                                              uint64_t seed) {
    const U4 d = draw(g, 0, kChance, seed);
    const int c0 = (int)pick(d.x, 3);
    const int j = (int)pick(d.y, 2);
    const int c1 = j + (j >= c0 ? 1 : 0);
    const int sd = c0 > c1 ? 1 : -1;
    const float u0 = u24(draw(g, 0, 0, seed).x);
    const float u1 = u24(draw(g, 1, 1, seed).x);
    const float u2 = u24(draw(g, 2, 0, seed).x);
    KuhnHand h;
    h.p[0] = tab6(t0, c0 * 2);                                  // seat 0 opens: P(bet)
    h.act[0] = u0 < h.p[0] ? 1 : 0;
    h.p[1] = tab6(t1, c1 * 2 + h.act[0]);                       // seat 1: P(bet) or P(call)
    h.act[1] = u1 < h.p[1] ? 1 : 0;
    h.p[2] = tab6(t0, c0 * 2 + 1);                              // seat 0 facing a bet: P(call)
    h.act[2] = u2 < h.p[2] ? 1 : 0;
    const bool third = h.act[0] == 0 && h.act[1] == 1;          // pass, bet
    h.n = third ? 3 : 2;
    h.payoff = h.act[0] ? (h.act[1] ? 2 * sd : 1)
                        : (h.act[1] ? (h.act[2] ? 2 * sd : -1) : sd);
    return h;
}

__global__ void __launch_bounds__(256) kuhn_eval_kernel(EvalArgs a) {
    const int pair = blockIdx.y;
    const int p0 = a.pairs[2 * pair], p1 = a.pairs[2 * pair + 1];
    const bool ok = pair_ok(a, p0, p1);
    if (!ok && threadIdx.x == 0 && blockIdx.x == 0) atomicOr(a.err, ERRBIT_BAD_PAIR);
    float t0[6], t1[6];
#pragma unroll
    for (int i = 0; i < 6; ++i) {
        t0[i] = ok ? a.arena[a.pol_offset[p0] + i] : 0.f;
        t1[i] = ok ? a.arena[a.pol_offset[p1] + i] : 0.f;
    }
    long long s1 = 0, s2 = 0, nd = 0;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    const int64_t n_play = ok ? a.n_episodes : 0;
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < n_play; e += stride) {
        const uint64_t g = (uint64_t)pair * (uint64_t)a.n_episodes + (uint64_t)e;
        const KuhnHand h = kuhn_play(t0, t1, g, a.seed);
        s1 += h.payoff;
        s2 += (long long)h.payoff * h.payoff;
        nd += h.n;
        if (e < a.n_dump) {
            const int64_t base = ((int64_t)pair * a.n_dump + e) * 3;
            for (int t = 0; t < 3; ++t) {
                const bool on = t < h.n;
                if (a.d_action) a.d_action[base + t] = on ? (uint8_t)h.act[t] : (uint8_t)255;
                if (a.d_reward) a.d_reward[base + t] = (t == h.n - 1) ? (float)h.payoff : 0.f;
                if (a.d_done) a.d_done[base + t] = (t >= h.n - 1) ? 1 : 0;
                if (a.d_logits) {
                    a.d_logits[(base + t) * 2] = on ? 1.f - h.p[t] : 0.f;
                    a.d_logits[(base + t) * 2 + 1] = on ? h.p[t] : 0.f;
                }
            }
        }
    }
    block_add_sums(s1, s2, nd, a.acc + 2 * pair, a.n_dec);
    // the pair's last block to finish writes its table row (its sums are final:
    // every block fenced its additions before counting itself)
    if (a.fin_out && threadIdx.x == 0) {
        __threadfence();
        if (atomicAdd(a.work + pair, 1ull) == (unsigned long long)gridDim.x - 1ull) {
            __threadfence();
            const long long f1 = (long long)__ldcg(a.acc + 2 * pair);
            const long long f2 = (long long)__ldcg(a.acc + 2 * pair + 1);
            finalize_pair(f1, f2, a.n_episodes, a.fin_out + 4 * (int64_t)pair);
        }
    }
}

// Exact expected seat-0 payoff: the 6 deals, each 1/6, times the betting tree.
__global__ void kuhn_exact_kernel(EvalArgs a, double* out) {
    const int pair = blockIdx.x * blockDim.x + threadIdx.x;
    if (pair >= a.n_pairs) return;
    const int p0 = a.pairs[2 * pair], p1 = a.pairs[2 * pair + 1];
    double v = 0.0;
    if (!pair_ok(a, p0, p1)) {
        atomicOr(a.err, ERRBIT_BAD_PAIR);
        v = __longlong_as_double(0x7ff8000000000000ll);
    } else {
        const float* t0 = a.arena + a.pol_offset[p0];
        const float* t1 = a.arena + a.pol_offset[p1];
        for (int c0 = 0; c0 < 3; ++c0)
            for (int c1 = 0; c1 < 3; ++c1) {
                if (c0 == c1) continue;
                const double sd = c0 > c1 ? 1.0 : -1.0;
                const double pb = t0[c0 * 2], pc = t1[c1 * 2 + 1];
                const double qb = t1[c1 * 2], qc = t0[c0 * 2 + 1];
                const double bet = pc * 2.0 * sd + (1.0 - pc);
                const double chk = (1.0 - qb) * sd + qb * (qc * 2.0 * sd - (1.0 - qc));
                v += (pb * bet + (1.0 - pb) * chk) / 6.0;
            }
    }
    out[4 * pair + 0] = v;
    out[4 * pair + 1] = 0.0;
    out[4 * pair + 2] = 0.0;
    out[4 * pair + 3] = 0.0;
}

constexpr int kLeducSlots = 248;      // hands in flight per CTA
constexpr int kLeducRowsMax = 256;    // 4-aligned seat-0 rows + 4-aligned seat-1 rows
constexpr int kLeducMaxDec = 8;

template <int H>
struct LeducF32Smem {
    using M = MlpF32<17, H, 3>;
    using L = typename M::L;
    static constexpr int kW = 0;
    static constexpr int kX = kW + 2 * L::kSize;
    static constexpr int kH1 = kX + kLeducRowsMax * M::XS;
    static constexpr int kLG = kH1 + M::kRowsPerPass * M::HS;
    static constexpr int kFloats = kLG + kLeducRowsMax * M::LS;
    static constexpr size_t kBytes = (size_t)kFloats * 4;
    static_assert(kLeducRowsMax % M::kRowsPerPass == 0, "rows tile the passes");
};

template <int H>
__global__ void __launch_bounds__(256, 1) leduc_eval_f32_kernel(EvalArgs a) {
    using SM = LeducF32Smem<H>;
    using M = typename SM::M;
    using L = typename SM::L;
    extern __shared__ __align__(128) float smem[];
    float* Ws = smem + SM::kW;
    float* X = smem + SM::kX;
    float* H1 = smem + SM::kH1;
    float* LG = smem + SM::kLG;
    __shared__ __align__(8) uint64_t bar;
    __shared__ int cnt[2][8];
    __shared__ unsigned long long next_e;

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    for (int i = tid; i < kLeducRowsMax * M::XS; i += blockDim.x) X[i] = 0.f;
    if (tid == 0) mbar_init(&bar, 1);
    __syncthreads();
    uint32_t parity = 0;

    const int64_t total = (int64_t)a.n_pairs * a.n_episodes;
    const int64_t per = (total + gridDim.x - 1) / gridDim.x;
    const int64_t lo = (int64_t)blockIdx.x * per;
    const int64_t hi = min(total, lo + per);

    for (int64_t seg = lo; seg < hi;) {
        const int pair = (int)(seg / a.n_episodes);
        const int64_t e_lo = seg - (int64_t)pair * a.n_episodes;
        const int64_t e_hi = min(a.n_episodes, e_lo + (hi - seg));
        seg += e_hi - e_lo;
        const int p0 = a.pairs[2 * pair], p1 = a.pairs[2 * pair + 1];
        if (!pair_ok(a, p0, p1)) {
            if (tid == 0) atomicOr(a.err, ERRBIT_BAD_PAIR);
            continue;
        }
        // stage the two policies (seat 0 at Ws, seat 1 at Ws + kSize)
        if (tid == 0) {
            fence_proxy_async_smem();
            mbar_arrive_expect_tx(&bar, 2u * L::kSize * 4u);
            for (int s = 0; s < 2; ++s) {
                const float* src = a.arena + a.pol_offset[s == 0 ? p0 : p1];
                for (uint32_t off = 0; off < (uint32_t)L::kSize * 4u; off += 32768u) {
                    const uint32_t n = min(32768u, (uint32_t)L::kSize * 4u - off);
                    bulk_g2s((char*)(Ws + s * L::kSize) + off, (const char*)src + off, n, &bar);
                }
            }
        }
        if (!mbar_wait_bounded(&bar, parity, kWaitLimitNs)) {
            if (tid == 0) atomicOr(a.err, ERRBIT_TIMEOUT);
            mbar_wait_bounded(&bar, parity, kWaitLimitNs);
            return;
        }
        parity ^= 1u;

        // hand slots
        LeducHand h;
        bool live = false;
        int64_t e = e_lo + tid;
        uint64_t g = 0;
        int t = 0;
        long long s1 = 0, s2 = 0, nd = 0;
        if (tid < kLeducSlots && e < e_hi) {
            live = true;
            g = (uint64_t)pair * (uint64_t)a.n_episodes + (uint64_t)e;
            leduc_deal(h, g, a.seed);
        }
        if (tid == 0) next_e = (unsigned long long)(e_lo + kLeducSlots);

        while (true) {
            const int seat = live ? h.actor : -1;
            const unsigned b0 = __ballot_sync(0xffffffffu, seat == 0);
            const unsigned b1 = __ballot_sync(0xffffffffu, seat == 1);
            if (lane == 0) { cnt[0][warp] = __popc(b0); cnt[1][warp] = __popc(b1); }
            __syncthreads();
            int n0 = 0, n1 = 0, pre0 = 0, pre1 = 0;
#pragma unroll
            for (int w = 0; w < 8; ++w) {
                const int x0 = cnt[0][w], x1 = cnt[1][w];
                if (w < warp) { pre0 += x0; pre1 += x1; }
                n0 += x0; n1 += x1;
            }
            if (n0 + n1 == 0) break;
            const int base1 = (n0 + 3) & ~3;
            const int rows = base1 + ((n1 + 3) & ~3);
            const unsigned lt = (1u << lane) - 1u;
            const int row = seat == 0 ? pre0 + __popc(b0 & lt) : base1 + pre1 + __popc(b1 & lt);
            float ob[17];
            if (live) {
                leduc_obs(h, ob);
                float* xr = X + row * M::XS;
#pragma unroll
                for (int i = 0; i < 17; ++i) xr[i] = ob[i];
            }
            __syncthreads();
            for (int r0 = 0; r0 < rows; r0 += M::kRowsPerPass) {
                const int grp = r0 + M::row_group() * 4;
                const float* w = grp < base1 ? Ws : Ws + L::kSize;
                M::pass(X, H1, LG, w, r0, r0 + M::warp_first_row() < rows);
            }
            if (live) {
                float lg[3] = {LG[row * M::LS], LG[row * M::LS + 1], LG[row * M::LS + 2]};
                const unsigned legal = leduc_legal(h);
                const float u = u24(draw(g, (uint32_t)t, (uint32_t)seat, a.seed).x);
                const int act = sample_masked<3>(lg, legal, u);
                const bool rec = e < a.n_dump;
                const int64_t rb = ((int64_t)pair * a.n_dump + e) * kLeducMaxDec;
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
                        for (int k = t; k < kLeducMaxDec; ++k) {
                            if (a.d_obs)
                                for (int i = 0; i < 20; ++i) a.d_obs[(rb + k) * 20 + i] = 0.f;
                            if (a.d_logits)
                                for (int i = 0; i < 3; ++i) a.d_logits[(rb + k) * 3 + i] = 0.f;
                            if (a.d_action) a.d_action[rb + k] = 255;
                            if (a.d_reward) a.d_reward[rb + k] = 0.f;
                            if (a.d_done) a.d_done[rb + k] = 1;
                        }
                    }
                    e = (int64_t)atomicAdd(&next_e, 1ull);
                    live = e < e_hi;
                    if (live) {
                        g = (uint64_t)pair * (uint64_t)a.n_episodes + (uint64_t)e;
                        leduc_deal(h, g, a.seed);
                        t = 0;
                    }
                }
            }
            __syncthreads();
        }
        block_add_sums(s1, s2, nd, a.acc + 2 * pair, a.n_dec);
    }
}


// Seat-phased Leduc evaluation for H = 128 (8x8 register tiles). Each step runs
// two 128-row passes, one per acting seat. Only one seat's W2 (64 KB) is
// resident; the small layers (W1, biases, W3) of both seats stay resident. The
// seat order alternates each step, so W2 is restaged once per step by bulk copy,
// overlapped with the second seat's layer 1. A seat with more than 128 acting
// hands defers the rest to the next step (their results do not depend on it).
//
// Work distribution: every pair has a hand counter in global memory shared by
// all CTAs that work on it. A CTA claims hands in chunks of kChunk and refills
// its slots from them; when the pair has no unclaimed hands left and its own
// hands have finished, it moves to the pair with the most unclaimed hands.
// Games differ in length from pair to pair, so a fixed split of the hands
// leaves CTAs with different numbers of steps; claiming keeps them finishing
// together. A hand's result depends only on its (pair, hand) ids, so the
// payoff sums do not depend on which CTA plays it.
namespace t8 {
using E = MlpF32T8<17, 3>;
using L = F32Layout<17, 128, 3>;
constexpr int kSlots = 248;
constexpr int kChunk = 128;                                   // hands per claim
constexpr int kRing = 8;                                      // claimed chunk starts kept
// at a step's start the unconsumed claimed chunks number at most kSlots / kChunk + 2
static_assert(kRing >= kSlots / kChunk + 3, "ring holds every chunk not yet handed out");
constexpr int kSmall = L::kW2T + (L::kSize - L::kB2);        // W1T|b1 then b2|W3|b3
constexpr int kOffSmall = 0;
constexpr int kOffW2 = kOffSmall + 2 * kSmall;
constexpr int kOffX = kOffW2 + 128 * 128;
constexpr int kOffH1 = kOffX + 2 * E::kRows * E::XS;
constexpr int kOffLG = kOffH1 + E::kRows * E::HS;
constexpr int kFloats = kOffLG + 2 * E::kRows * E::LS;
constexpr size_t kBytes = (size_t)kFloats * 4;
static_assert(kSmall % 4 == 0 && kOffW2 % 4 == 0 && kOffX % 4 == 0 && kOffH1 % 4 == 0, "16-B");

struct Claims {
    unsigned long long next;      // next slot number to hand out in this segment
    unsigned long long n;         // chunks claimed in this segment
    long long base[kRing];        // first hand of chunk c at base[c % kRing]
    int done;                     // the pair has no unclaimed hands left
};

// One thread: claim chunks until slots [next, next + kSlots) are covered.
__device__ __forceinline__ void top_up(Claims& c, unsigned long long* counter, int64_t n_episodes) {
    while (!c.done && c.n * kChunk < c.next + kSlots) {
        const unsigned long long s = atomicAdd(counter, (unsigned long long)kChunk);
        if (s >= (unsigned long long)n_episodes) { c.done = 1; break; }
        c.base[c.n % kRing] = (long long)s;
        ++c.n;
        if (s + kChunk >= (unsigned long long)n_episodes) c.done = 1;
    }
}

// Hand of slot j, or -1 when the pair has none left for it.
__device__ __forceinline__ int64_t slot_hand(const Claims& c, unsigned long long j, int64_t n_episodes) {
    const unsigned long long ch = j / kChunk;
    if (ch >= c.n) return -1;
    const int64_t e = c.base[ch % kRing] + (int64_t)(j % kChunk);
    return e < n_episodes ? e : -1;
}

// All threads: the pair with the most unclaimed hands (-1 when none has any).
// Ends with a barrier; the result is uniform across the CTA.
__device__ int pick_pair(const EvalArgs& a) {
    __shared__ long long rem_w[8];
    __shared__ int pair_w[8];
    long long best = 0;
    int bp = -1;
    for (int p = threadIdx.x; p < a.n_pairs; p += blockDim.x) {
        const unsigned long long w = *reinterpret_cast<volatile unsigned long long*>(a.work + p);
        const long long rem = w >= (unsigned long long)a.n_episodes ? 0 : a.n_episodes - (long long)w;
        if (rem > best) { best = rem; bp = p; }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const long long ob = __shfl_xor_sync(0xffffffffu, best, o);
        const int op = __shfl_xor_sync(0xffffffffu, bp, o);
        if (ob > best || (ob == best && op >= 0 && (bp < 0 || op < bp))) { best = ob; bp = op; }
    }
    const int warp = threadIdx.x >> 5;
    if ((threadIdx.x & 31) == 0) { rem_w[warp] = best; pair_w[warp] = bp; }
    __syncthreads();
    best = 0;
    bp = -1;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w)
        if (rem_w[w] > best) { best = rem_w[w]; bp = pair_w[w]; }
    __syncthreads();
    return bp;
}
// 16-row blocks a pass of c placed rows (compacted into rows 0 .. c - 1)
// computes: ceil(c / 16), at least 4.
__device__ __forceinline__ int blocks_for(int c) { return c <= 64 ? 4 : (c + 15) >> 4; }

template <class Eng>
__device__ __forceinline__ void layer1_n(int nb, const float* X, float* H1, const float* W1T,
                                         const float* b1) {
    switch (nb) {
        case 4: Eng::template layer1<4>(X, H1, W1T, b1); break;
        case 5: Eng::template layer1<5>(X, H1, W1T, b1); break;
        case 6: Eng::template layer1<6>(X, H1, W1T, b1); break;
        case 7: Eng::template layer1<7>(X, H1, W1T, b1); break;
        default: Eng::template layer1<8>(X, H1, W1T, b1); break;
    }
}

template <class Eng>
__device__ __forceinline__ void layer23_n(int nb, const float* H1, float* LG, const float* W2T,
                                          const float* b2, const float* W3, const float* b3) {
    switch (nb) {
        case 4: Eng::template layer23<4>(H1, LG, W2T, b2, W3, b3); break;
        case 5: Eng::template layer23<5>(H1, LG, W2T, b2, W3, b3); break;
        case 6: Eng::template layer23<6>(H1, LG, W2T, b2, W3, b3); break;
        case 7: Eng::template layer23<7>(H1, LG, W2T, b2, W3, b3); break;
        default: Eng::template layer23<8>(H1, LG, W2T, b2, W3, b3); break;
    }
}

}  // namespace t8

// kDump: the call records its first n_dump hands of every pair (the recording
// code is compiled out of the other instance).
template <bool kDump>
__global__ void __launch_bounds__(256, 1) leduc_eval_f32_t8_kernel(EvalArgs a) {
    using namespace t8;
    extern __shared__ __align__(128) float smem[];
    float* X = smem + kOffX;
    float* H1 = smem + kOffH1;
    float* LG = smem + kOffLG;
    float* W2s = smem + kOffW2;
    __shared__ __align__(8) uint64_t bar;
    __shared__ int cnt[2][8];
    __shared__ Claims cl;

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    for (int i = tid; i < 2 * E::kRows * E::XS; i += blockDim.x) X[i] = 0.f;
    if (tid == 0) mbar_init(&bar, 1);
    __syncthreads();
    uint32_t parity = 0;

    int pair = (int)(((int64_t)blockIdx.x * a.n_pairs) / gridDim.x);
    while (pair >= 0) {
        unsigned long long* counter = a.work + pair;
        const int pid[2] = {a.pairs[2 * pair], a.pairs[2 * pair + 1]};
        if (!pair_ok(a, pid[0], pid[1])) {
            if (tid == 0) {
                atomicOr(a.err, ERRBIT_BAD_PAIR);
                atomicMax(counter, (unsigned long long)a.n_episodes);
            }
            pair = pick_pair(a);
            continue;
        }
        const float* pol0 = a.arena + a.pol_offset[pid[0]];
        const float* pol1 = a.arena + a.pol_offset[pid[1]];
        int res = 0;                                    // seat whose W2 is resident
        if (tid == 0) {
            fence_proxy_async_smem();
            mbar_arrive_expect_tx(&bar, 2u * kSmall * 4u + 128u * 128u * 4u);
            for (int s = 0; s < 2; ++s) {
                const float* src = s == 0 ? pol0 : pol1;
                float* dst = smem + kOffSmall + s * kSmall;
                bulk_g2s(dst, src, L::kW2T * 4u, &bar);
                bulk_g2s(dst + L::kW2T, src + L::kB2, (L::kSize - L::kB2) * 4u, &bar);
            }
            bulk_g2s(W2s, pol0 + L::kW2T, 32768u, &bar);
            bulk_g2s(W2s + 8192, pol0 + L::kW2T + 8192, 32768u, &bar);
            cl.next = 0;
            cl.n = 0;
            cl.done = 0;
            top_up(cl, counter, a.n_episodes);
            cl.next = kSlots;                           // slots 0..kSlots-1 go to threads 0..kSlots-1
        }
        if (!mbar_wait_bounded(&bar, parity, kWaitLimitNs) && tid == 0) atomicOr(a.err, ERRBIT_TIMEOUT);
        parity ^= 1u;
        __syncthreads();

        LeducHand h;
        bool live = false;
        int64_t e = tid < kSlots ? slot_hand(cl, (unsigned long long)tid, a.n_episodes) : -1;
        uint64_t g = 0;
        int t = 0;
        long long s1 = 0, s2 = 0, nd = 0;
        if (e >= 0) {
            live = true;
            g = (uint64_t)pair * (uint64_t)a.n_episodes + (uint64_t)e;
            leduc_deal(h, g, a.seed);
        }

        while (true) {
            // claims for this step's refills; every reader of cl passed the last barrier
            if (tid == 0) top_up(cl, counter, a.n_episodes);
            const int seat = live ? h.actor : -1;
            const unsigned b0 = __ballot_sync(0xffffffffu, seat == 0);
            const unsigned b1 = __ballot_sync(0xffffffffu, seat == 1);
            if (lane == 0) { cnt[0][warp] = __popc(b0); cnt[1][warp] = __popc(b1); }
            __syncthreads();
            int c[2] = {0, 0}, pre = 0;
#pragma unroll
            for (int w = 0; w < 8; ++w) {
                c[0] += cnt[0][w];
                c[1] += cnt[1][w];
                if (w < warp) pre += seat == 1 ? cnt[1][w] : cnt[0][w];
            }
            if (c[0] + c[1] == 0) break;
            const unsigned mine = seat == 1 ? b1 : b0;
            const int rank = pre + __popc(mine & ((1u << lane) - 1u));
            const bool placed = live && rank < E::kRows;
            float ob[17];
            if (placed) {
                leduc_obs(h, ob);
                float* xr = X + (seat * E::kRows + rank) * E::XS;
#pragma unroll
                for (int i = 0; i < 17; ++i) xr[i] = ob[i];
            }
            __syncthreads();
            const int first = res, second = 1 - res;
            const float* sf = smem + kOffSmall + first * kSmall;
            const float* ss = smem + kOffSmall + second * kSmall;
            const int off_b2 = L::kW2T, off_w3 = L::kW2T + (L::kW3 - L::kB2),
                      off_b3 = L::kW2T + (L::kB3 - L::kB2);
            // a pass computes the 16-row blocks that hold its placed rows (at
            // least 4)
            if (c[first] > 0) {
                const int nb = t8::blocks_for(c[first]);
                t8::layer1_n<E>(nb, X + first * E::kRows * E::XS, H1, sf, sf + L::kB1);
                t8::layer23_n<E>(nb, H1, LG + first * E::kRows * E::LS, W2s, sf + off_b2, sf + off_w3,
                                 sf + off_b3);
            }
            if (c[second] > 0) {
                const float* src = (second == 0 ? pol0 : pol1) + L::kW2T;
                if (tid == 0) {                       // every read of W2s has passed a barrier
                    fence_proxy_async_smem();
                    mbar_arrive_expect_tx(&bar, 128u * 128u * 4u);
                    bulk_g2s(W2s, src, 32768u, &bar);
                    bulk_g2s(W2s + 8192, src + 8192, 32768u, &bar);
                }
                const int nb = t8::blocks_for(c[second]);
                t8::layer1_n<E>(nb, X + second * E::kRows * E::XS, H1, ss, ss + L::kB1);
                if (!mbar_wait_bounded(&bar, parity, kWaitLimitNs) && tid == 0)
                    atomicOr(a.err, ERRBIT_TIMEOUT);
                parity ^= 1u;
                t8::layer23_n<E>(nb, H1, LG + second * E::kRows * E::LS, W2s, ss + off_b2, ss + off_w3,
                                 ss + off_b3);
                res = second;
            }
            if (placed) {
                const float* lp = LG + (seat * E::kRows + rank) * E::LS;
                float lg[3] = {lp[0], lp[1], lp[2]};
                const unsigned legal = leduc_legal(h);
                const float u = u24(draw(g, (uint32_t)t, (uint32_t)seat, a.seed).x);
                const int act = sample_masked<3>(lg, legal, u);
                const bool rec = kDump && e < a.n_dump;
                const int64_t rb = ((int64_t)pair * a.n_dump + e) * kLeducMaxDec;
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
                        for (int k = t; k < kLeducMaxDec; ++k) {
                            if (a.d_obs)
                                for (int i = 0; i < 20; ++i) a.d_obs[(rb + k) * 20 + i] = 0.f;
                            if (a.d_logits)
                                for (int i = 0; i < 3; ++i) a.d_logits[(rb + k) * 3 + i] = 0.f;
                            if (a.d_action) a.d_action[rb + k] = 255;
                            if (a.d_reward) a.d_reward[rb + k] = 0.f;
                            if (a.d_done) a.d_done[rb + k] = 1;
                        }
                    }
                    e = slot_hand(cl, atomicAdd(&cl.next, 1ull), a.n_episodes);
                    live = e >= 0;
                    if (live) {
                        g = (uint64_t)pair * (uint64_t)a.n_episodes + (uint64_t)e;
                        leduc_deal(h, g, a.seed);
                        t = 0;
                    }
                }
            }
            __syncthreads();
        }
        block_add_sums(s1, s2, nd, a.acc + 2 * pair, a.n_dec);
        pair = pick_pair(a);
    }
}

}  // namespace

bool leduc_f32_supported(int hidden) { return hidden == 128 || hidden == 64; }

cudaError_t launch_kuhn_eval(const EvalArgs& a, int n_sm, cudaStream_t s) {
    if (a.n_pairs == 0) return cudaSuccess;
    int64_t blocks_per_pair = (a.n_episodes + 255) / 256;
    const int64_t cap = max(1, (n_sm * 8) / max(1, a.n_pairs));
    if (blocks_per_pair > cap) blocks_per_pair = cap;
    if (blocks_per_pair > 65535) blocks_per_pair = 65535;
    dim3 grid((unsigned)blocks_per_pair, (unsigned)a.n_pairs);
    kuhn_eval_kernel<<<grid, 256, 0, s>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_kuhn_exact(const EvalArgs& a, double* out, cudaStream_t s) {
    if (a.n_pairs == 0) return cudaSuccess;
    kuhn_exact_kernel<<<(a.n_pairs + 127) / 128, 128, 0, s>>>(a, out);
    return cudaGetLastError();
}

template <int H>
static cudaError_t launch_leduc_h(const EvalArgs& a, int n_sm, cudaStream_t s) {
    const size_t bytes = LeducF32Smem<H>::kBytes;
    cudaError_t err = cudaFuncSetAttribute(leduc_eval_f32_kernel<H>,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
    if (err != cudaSuccess) return err;
    const int64_t total = (int64_t)a.n_pairs * a.n_episodes;
    int64_t grid = (total + kLeducSlots - 1) / kLeducSlots;
    if (grid > n_sm) grid = n_sm;
    if (grid < 1) grid = 1;
    leduc_eval_f32_kernel<H><<<(unsigned)grid, 256, bytes, s>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_leduc_eval_f32(const EvalArgs& a, int hidden, int n_sm, cudaStream_t s) {
    if (a.n_pairs == 0) return cudaSuccess;
    if (hidden == 128) {
        if (!a.work) return cudaErrorInvalidValue;       // the kernel claims hands from a.work
        auto kern = a.n_dump > 0 ? leduc_eval_f32_t8_kernel<true> : leduc_eval_f32_t8_kernel<false>;
        cudaError_t err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               (int)t8::kBytes);
        if (err != cudaSuccess) return err;
        const int64_t total = (int64_t)a.n_pairs * a.n_episodes;
        int64_t grid = (total + t8::kSlots - 1) / t8::kSlots;
        if (grid > n_sm) grid = n_sm;
        if (grid < 1) grid = 1;
        kern<<<(unsigned)grid, 256, t8::kBytes, s>>>(a);
        return cudaGetLastError();
    }
    if (hidden == 64) return launch_leduc_h<64>(a, n_sm, s);
    return cudaErrorInvalidValue;
}

}  // namespace malib
