// CPU oracle for the MALib (arXiv 2106.07551) rollout / payoff-evaluation path.
//
// TEST INFRASTRUCTURE ONLY. This is a plain, slow, obviously-correct CPU
// restatement of what the GPU path computes, used to check it. Only the test
// suite, the smoke check and the CPU-baseline leg of the benchmark may load it.
// It shares no source with the CUDA path (no header, no helper, no table).
//
// What it follows:
//  * Sec. 3.1 "Defining the Task Graph": a population of policy pools, one
//    policy per agent forms a combination Comb_t; a rollout draws
//    X ~ P(s, a, s' | a ~ Comb_t).
//  * Sec. 3.2: the Evaluator keeps a payoff table with one entry per policy
//    combination; Sec. 4.2 (Leduc PSRO): each entry is the Monte-Carlo mean over
//    a fixed number of simulations of that combination.
//  * App. B.1 "Simple Spread": N agents cover N landmarks; reward is minus the
//    sum over landmarks of the distance to the closest agent, minus one per
//    collision.
//  * App. B.1 "Simple Speaker Listener": a speaker that cannot move sends one of
//    three messages naming the target landmark; the listener, which cannot
//    speak, navigates to it; both are rewarded by the listener's distance.
//  * App. B.1 "Simple Adversary": one adversary and two good agents, two
//    landmarks of which one is the target; good agents are rewarded for being
//    close to the target and for the adversary being far from it, the adversary
//    (which is not told the target) for being close to it.
//  * App. B.1 "Simple Push": one good agent, one adversary, one landmark; the
//    good agent is rewarded by its distance to the landmark, the adversary by
//    the difference of the two distances, so it learns to push.
//  * App. B.1 "Simple Tag": one faster good agent, three slower adversaries,
//    two obstacles that block the way; -10 to the good agent and +10 to the
//    adversaries for each hit.
//  * App. B.1 "Simple Reference": two agents that each know only the other's
//    goal landmark, both speaking and moving, rewarded by their own distance
//    and the average distance, weighted by local_ratio.
//  * Collisions of App. B.1 as forces (push, tag, and spread as an option): a
//    soft contact model between disks, a stated reading (the paper gives no
//    force law).
// Kuhn and Leduc rules are not given in the paper; the textbook rules are used,
// each reading stated at the function that takes it below.
//
// Numerics: fp32 where the method is defined in fp32 (environment dynamics,
// sampling); policy forward accumulated in fp64 and rounded to fp32 logits;
// bf16 policies round weights and every layer's input to bf16 first. Compiled
// with -ffp-contract=off so that no multiply-add is fused behind our back.
//
// Parity status: Philox, det_expf, Kuhn (exact enumeration), Leduc (tree
// enumeration, hand-worked hands), spread (closed-form single steps and
// invariants), the simple adversary (hand-worked geometry, the reward
// identity against fp64, the spread dynamics and reset, symmetries) and the
// simple speaker listener (hand-worked geometry, the one-step message delay,
// the immobile speaker, the spread dynamics and reset, the target draw), the
// contact model (log1p against the library, the force against its formula in
// fp64, zero beyond the margin, equal and opposite pairs, total velocity
// against the closed form), simple push (hand-worked geometry, contact on both
// agents) and simple tag (speed limits against the capped recursion, the hit
// rule, immovable obstacles, the observation layout) and simple reference
// (hand-worked rewards, the message delay, the moves against spread, the goal
// draws) are pinned by the CPU tests, and whole spread episodes under forced actions (at
// rest; a constant force from rest) match closed forms; episode returns of the
// particle scenarios under sampled policies beyond those are "parity unpinned"
// (no closed form exists).

#include <algorithm>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <thread>
#include <vector>

namespace {

// ---------------------------------------------------------------------------
// Philox4x32-10 (Salmon, Moraes, Dror, Shaw, "Parallel random numbers: as easy
// as 1, 2, 3", SC'11). Counter (c0..c3), key (k0, k1) = (seed lo, seed hi).
// Each round: two 32x32->64 products of c0 and c2 with the round multipliers,
// the high halves xored with the other two words and the key; the key is
// bumped by the Weyl constants between rounds.
// ---------------------------------------------------------------------------
struct Words { uint32_t x[4]; };

Words philox4x32_10(uint32_t c0, uint32_t c1, uint32_t c2, uint32_t c3, uint64_t seed) {
    const uint32_t M0 = 0xD2511F53u, M1 = 0xCD9E8D57u;
    const uint32_t W0 = 0x9E3779B9u, W1 = 0xBB67AE85u;
    uint32_t k0 = (uint32_t)(seed & 0xFFFFFFFFu);
    uint32_t k1 = (uint32_t)(seed >> 32);
    uint32_t c[4] = {c0, c1, c2, c3};
    for (int round = 0; round < 10; ++round) {
        if (round > 0) { k0 += W0; k1 += W1; }
        uint64_t prod0 = (uint64_t)M0 * (uint64_t)c[0];
        uint64_t prod1 = (uint64_t)M1 * (uint64_t)c[2];
        uint32_t hi0 = (uint32_t)(prod0 >> 32), lo0 = (uint32_t)prod0;
        uint32_t hi1 = (uint32_t)(prod1 >> 32), lo1 = (uint32_t)prod1;
        uint32_t n0 = hi1 ^ c[1] ^ k0;
        uint32_t n1 = lo1;
        uint32_t n2 = hi0 ^ c[3] ^ k1;
        uint32_t n3 = lo0;
        c[0] = n0; c[1] = n1; c[2] = n2; c[3] = n3;
    }
    Words w;
    for (int i = 0; i < 4; ++i) w.x[i] = c[i];
    return w;
}

// Counter layout (reading of "keyed by (seed, env, step, agent)"):
//   (g lo32, g hi32, step, agent); g = global episode id.
// Chance draws use agent = 0xFFFFFFFF; for spread resets the step field holds
// the entity (agent i -> i, landmark l -> 0x80000000 + l).
const uint32_t CHANCE = 0xFFFFFFFFu;

Words draw(uint64_t g, uint32_t step, uint32_t agent, uint64_t seed) {
    return philox4x32_10((uint32_t)(g & 0xFFFFFFFFu), (uint32_t)(g >> 32), step, agent, seed);
}

// Uniform in [0, 1): the top 24 bits of a word times 2^-24 (exact in fp32).
float uniform24(uint32_t x) { return (float)(x >> 8) * 5.9604644775390625e-08f; }

// Index in [0, n) from a word: multiply-shift (Lemire), (x * n) >> 32.
uint32_t pick(uint32_t x, uint32_t n) { return (uint32_t)(((uint64_t)x * (uint64_t)n) >> 32); }

// ---------------------------------------------------------------------------
// det_expf: exp(x) in fp32 whose every step is a correctly-rounded IEEE
// operation, so that two implementations of the same steps agree bit for bit.
// Method: Cody-Waite argument reduction x = k ln2 + r with ln2 split into a
// short head (exact products k*head) and a tail; exp(r) by the Taylor series
// to degree 7 in Horner form with fused multiply-adds; 2^k applied by building
// the power of two from its exponent field. Inputs at or below -87 give 0.
// ---------------------------------------------------------------------------
float det_expf(float x) {
    if (!(x > -87.0f)) return 0.0f;
    if (x > 88.0f) x = 88.0f;
    const float LOG2E = 0x1.715476p+0f;
    const float LN2_HEAD = 0x1.62e4p-1f;
    const float LN2_TAIL = 0x1.7f7d1cp-20f;
    float kf = rintf(x * LOG2E);
    float r = fmaf(-kf, LN2_HEAD, x);
    r = fmaf(-kf, LN2_TAIL, r);
    float p = 0x1.a01a02p-13f;        // 1/7!
    p = fmaf(p, r, 0x1.6c16c2p-10f);  // 1/6!
    p = fmaf(p, r, 0x1.111112p-7f);   // 1/5!
    p = fmaf(p, r, 0x1.555556p-5f);   // 1/4!
    p = fmaf(p, r, 0x1.555556p-3f);   // 1/3!
    p = fmaf(p, r, 0.5f);             // 1/2!
    p = fmaf(p, r, 1.0f);
    p = fmaf(p, r, 1.0f);
    int k = (int)kf;                  // in [-126, 127] for the clamped domain
    uint32_t bits = (uint32_t)(k + 127) << 23;
    float two_k;
    std::memcpy(&two_k, &bits, 4);
    return p * two_k;
}

// Masked softmax + inverse-CDF draw, no division:
//   m = max over legal logits; e_a = det_expf(l_a - m) for legal a, 0 otherwise;
//   S = sum of e_a in ascending a; the action is the first legal a whose
//   running sum C_a exceeds u*S; if rounding leaves none, the last legal a.
int sample_masked(const float* logits, const uint8_t* legal, int A, float u) {
    int first = -1;
    for (int a = 0; a < A; ++a) if (legal[a]) { first = a; break; }
    if (first < 0) return -1;
    float m = logits[first];
    for (int a = first + 1; a < A; ++a) if (legal[a] && logits[a] > m) m = logits[a];
    float e[16];
    float S = 0.0f;
    for (int a = 0; a < A; ++a) {
        e[a] = legal[a] ? det_expf(logits[a] - m) : 0.0f;
        S = S + e[a];
    }
    float thr = u * S;
    float C = 0.0f;
    int last = first;
    for (int a = 0; a < A; ++a) {
        if (!legal[a]) continue;
        C = C + e[a];
        last = a;
        if (thr < C) return a;
    }
    return last;
}

// bf16 round-to-nearest-even of an fp32 value (returned widened to fp32).
float bf16_round(float x) {
    uint32_t b;
    std::memcpy(&b, &x, 4);
    if ((b & 0x7F800000u) == 0x7F800000u) return x;  // inf / nan unchanged
    uint32_t lsb = (b >> 16) & 1u;
    b += 0x7FFFu + lsb;
    b &= 0xFFFF0000u;
    float y;
    std::memcpy(&y, &b, 4);
    return y;
}

// ---------------------------------------------------------------------------
// MLP policy forward: logits = W3 relu(W2 relu(W1 x + b1) + b2) + b3 with the
// parameter layout W1[h1][in], b1, W2[h2][h1], b2, W3[out][h2], b3. Sums in
// fp64, logits rounded once to fp32. bf16 policies: weights and each layer's
// input rounded to bf16 (the hidden layers via fp32).
// ---------------------------------------------------------------------------
struct Mlp {
    const float* p;
    int in, h1, h2, out;
    int bf16;
};

void mlp_logits(const Mlp& m, const float* x, float* logits) {
    const float* W1 = m.p;
    const float* b1 = W1 + (size_t)m.h1 * m.in;
    const float* W2 = b1 + m.h1;
    const float* b2 = W2 + (size_t)m.h2 * m.h1;
    const float* W3 = b2 + m.h2;
    const float* b3 = W3 + (size_t)m.out * m.h2;
    auto w = [&](float v) -> double { return m.bf16 ? (double)bf16_round(v) : (double)v; };
    auto act = [&](double v) -> double { return m.bf16 ? (double)bf16_round((float)v) : v; };
    std::vector<double> a0(m.in), a1(m.h1), a2(m.h2);
    for (int i = 0; i < m.in; ++i) a0[i] = m.bf16 ? (double)bf16_round(x[i]) : (double)x[i];
    for (int j = 0; j < m.h1; ++j) {
        double s = (double)b1[j];
        for (int i = 0; i < m.in; ++i) s += w(W1[(size_t)j * m.in + i]) * a0[i];
        a1[j] = act(s > 0.0 ? s : 0.0);
    }
    for (int j = 0; j < m.h2; ++j) {
        double s = (double)b2[j];
        for (int i = 0; i < m.h1; ++i) s += w(W2[(size_t)j * m.h1 + i]) * a1[i];
        a2[j] = act(s > 0.0 ? s : 0.0);
    }
    for (int j = 0; j < m.out; ++j) {
        double s = (double)b3[j];
        for (int i = 0; i < m.h2; ++i) s += w(W3[(size_t)j * m.h2 + i]) * a2[i];
        logits[j] = (float)s;
    }
}

int n_threads_or_default(int n) {
    if (n > 0) return n;
    unsigned h = std::thread::hardware_concurrency();
    return h ? (int)h : 1;
}

template <class F>
void parallel_for(int64_t n, int n_threads, F f) {
    n_threads = n_threads_or_default(n_threads);
    if (n_threads > n) n_threads = (int)std::max<int64_t>(n, 1);
    if (n_threads <= 1) { for (int64_t i = 0; i < n; ++i) f(i); return; }
    std::vector<std::thread> th;
    for (int t = 0; t < n_threads; ++t) {
        th.emplace_back([=]() { for (int64_t i = t; i < n; i += n_threads) f(i); });
    }
    for (auto& x : th) x.join();
}

// Payoff-table entry from integer sums: mean, standard error of the mean
// (sample variance with n-1; 0 when n < 2), sum, sum of squares.
void finish_entry(int64_t s1, int64_t s2, int64_t n, double* out4) {
    double mean = (double)s1 / (double)n;
    double se = 0.0;
    if (n >= 2) {
        double var = ((double)s2 - (double)s1 * (double)s1 / (double)n) / (double)(n - 1);
        if (var < 0.0) var = 0.0;
        se = std::sqrt(var / (double)n);
    }
    out4[0] = mean; out4[1] = se; out4[2] = (double)s1; out4[3] = (double)s2;
}

// ---------------------------------------------------------------------------
// Kuhn poker (textbook rules). Cards J=0 < Q=1 < K=2, ante 1 each, one bet of 1.
// Seat 0 passes or bets. pass-pass: showdown for 1. pass-bet: seat 0 calls
// (showdown for 2) or folds (-1). bet: seat 1 calls (showdown for 2) or folds
// (+1). A tabular policy gives P(bet) per infoset card*2 + h, h = 0 at the
// seat's first decision, h = 1 when facing a bet (there "bet" means call).
// ---------------------------------------------------------------------------
struct KuhnTrace { int card0, card1, n_dec; int seat[3], action[3]; float pbet[3]; int payoff0; };

int kuhn_episode(const float* pol0, const float* pol1, uint64_t g, uint64_t seed, KuhnTrace* tr) {
    Words d = draw(g, 0, CHANCE, seed);
    int deck[3] = {0, 1, 2};
    int i0 = (int)pick(d.x[0], 3);
    int c0 = deck[i0];
    int rest[2], r = 0;
    for (int i = 0; i < 3; ++i) if (i != i0) rest[r++] = deck[i];
    int c1 = rest[pick(d.x[1], 2)];
    int t = 0;
    int payoff;
    auto decide = [&](int seat, float p) -> int {
        float u = uniform24(draw(g, (uint32_t)t, (uint32_t)seat, seed).x[0]);
        int a = (u < p) ? 1 : 0;
        if (tr) { tr->seat[t] = seat; tr->action[t] = a; tr->pbet[t] = p; }
        ++t;
        return a;
    };
    int showdown = (c0 > c1) ? 1 : -1;
    if (decide(0, pol0[c0 * 2 + 0])) {            // seat 0 bets
        if (decide(1, pol1[c1 * 2 + 1])) payoff = 2 * showdown;  // seat 1 calls
        else payoff = 1;                                          // seat 1 folds
    } else {                                       // seat 0 passes
        if (decide(1, pol1[c1 * 2 + 0])) {         // seat 1 bets
            if (decide(0, pol0[c0 * 2 + 1])) payoff = 2 * showdown;  // seat 0 calls
            else payoff = -1;                                         // seat 0 folds
        } else {
            payoff = showdown;
        }
    }
    if (tr) { tr->card0 = c0; tr->card1 = c1; tr->n_dec = t; tr->payoff0 = payoff; }
    return payoff;
}

// Expected seat-0 payoff by enumerating the 6 deals (each 1/6) and the tree.
double kuhn_exact(const float* pol0, const float* pol1) {
    double total = 0.0;
    for (int c0 = 0; c0 < 3; ++c0) {
        for (int c1 = 0; c1 < 3; ++c1) {
            if (c0 == c1) continue;
            double sd = (c0 > c1) ? 1.0 : -1.0;
            double p = pol0[c0 * 2 + 0], q = pol1[c1 * 2 + 1];
            double rr = pol1[c1 * 2 + 0], s = pol0[c0 * 2 + 1];
            double v_bet = q * 2.0 * sd + (1.0 - q) * 1.0;
            double v_pass = (1.0 - rr) * sd + rr * (s * 2.0 * sd + (1.0 - s) * -1.0);
            total += (p * v_bet + (1.0 - p) * v_pass) / 6.0;
        }
    }
    return total;
}

// ---------------------------------------------------------------------------
// Leduc hold'em (readings of the standard game): 6 cards, two each of J, Q, K
// (card index c, rank c / 2); ante 1; two betting rounds with raise size 2
// then 4; at most 2 raises per round (the first bet counts); seat 0 acts first
// in both rounds; the public card is revealed after round 1. Fold is legal only
// when facing an outstanding bet, call (check) always, raise while fewer than 2
// raises this round. A round ends once both seats have acted and the
// contributions are equal. Showdown: pairing the public card wins, else the
// higher private rank, equal ranks split (payoff 0). The winner gains the
// loser's contribution.
// Actions: 0 fold, 1 call/check, 2 raise.
// ---------------------------------------------------------------------------
struct Leduc {
    int card[2];
    int pub;
    int round;        // 0 or 1
    int contrib[2];
    int raises;       // raises this round
    int n_act;        // actions taken this round
    int actor;
    int done;
    int payoff0;
};

void leduc_init(Leduc& s, int c0, int c1, int pub) {
    s.card[0] = c0; s.card[1] = c1; s.pub = pub;
    s.round = 0; s.contrib[0] = 1; s.contrib[1] = 1;
    s.raises = 0; s.n_act = 0; s.actor = 0; s.done = 0; s.payoff0 = 0;
}

void leduc_legal(const Leduc& s, uint8_t legal[3]) {
    int me = s.actor, opp = 1 - me;
    legal[0] = s.contrib[opp] > s.contrib[me] ? 1 : 0;
    legal[1] = 1;
    legal[2] = s.raises < 2 ? 1 : 0;
}

int leduc_showdown(const Leduc& s) {
    int r0 = s.card[0] / 2, r1 = s.card[1] / 2, rp = s.pub / 2;
    int win;   // +1 seat 0 wins, -1 seat 1 wins, 0 split
    if (r0 == rp) win = 1;
    else if (r1 == rp) win = -1;
    else if (r0 > r1) win = 1;
    else if (r1 > r0) win = -1;
    else win = 0;
    if (win > 0) return s.contrib[1];
    if (win < 0) return -s.contrib[0];
    return 0;
}

// Applies a legal action. Returns 0, or -1 if the action is illegal.
int leduc_apply(Leduc& s, int a) {
    uint8_t legal[3];
    leduc_legal(s, legal);
    if (a < 0 || a > 2 || !legal[a] || s.done) return -1;
    int me = s.actor, opp = 1 - me;
    if (a == 0) {
        s.done = 1;
        s.payoff0 = (me == 0) ? -s.contrib[0] : s.contrib[1];
        return 0;
    }
    s.n_act += 1;
    if (a == 2) {
        s.contrib[me] = s.contrib[opp] + (s.round == 0 ? 2 : 4);
        s.raises += 1;
        s.actor = opp;
        return 0;
    }
    s.contrib[me] = s.contrib[opp];
    if (s.n_act >= 2) {
        if (s.round == 0) {
            s.round = 1; s.raises = 0; s.n_act = 0; s.actor = 0;
        } else {
            s.done = 1;
            s.payoff0 = leduc_showdown(s);
        }
    } else {
        s.actor = opp;
    }
    return 0;
}

// Observation of the acting seat, 17 floats: private rank one-hot (J,Q,K),
// public rank one-hot (J,Q,K,none), round one-hot, own and opponent
// contribution / 13, raises-this-round one-hot (0,1,2), legal mask (f,c,r).
void leduc_obs(const Leduc& s, float* o) {
    for (int i = 0; i < 17; ++i) o[i] = 0.0f;
    int me = s.actor, opp = 1 - me;
    o[s.card[me] / 2] = 1.0f;
    o[3 + (s.round == 1 ? s.pub / 2 : 3)] = 1.0f;
    o[7 + s.round] = 1.0f;
    o[9] = (float)s.contrib[me] / 13.0f;
    o[10] = (float)s.contrib[opp] / 13.0f;
    o[11 + s.raises] = 1.0f;
    uint8_t legal[3];
    leduc_legal(s, legal);
    for (int a = 0; a < 3; ++a) o[14 + a] = legal[a] ? 1.0f : 0.0f;
}

// Deal: seat 0, seat 1, public, each drawn from the cards still in the deck
// in index order, from one chance draw.
void leduc_deal(uint64_t g, uint64_t seed, int* c0, int* c1, int* pub) {
    Words d = draw(g, 0, CHANCE, seed);
    std::vector<int> deck = {0, 1, 2, 3, 4, 5};
    int k = (int)pick(d.x[0], 6);
    *c0 = deck[k]; deck.erase(deck.begin() + k);
    k = (int)pick(d.x[1], 5);
    *c1 = deck[k]; deck.erase(deck.begin() + k);
    k = (int)pick(d.x[2], 4);
    *pub = deck[k];
}

const int LEDUC_MAX_DEC = 8;

struct DecisionRecord {   // per decision slot of a dumped episode
    float* obs;           // [obs_dim]
    float* logits;        // [A]
};

// One Leduc episode. ext (optional, [8][3]) replaces the oracle's own logits
// in the draw (replay of another implementation's logits); own logits, obs,
// actions, acting seats and the payoff are recorded when the pointers are set.
int leduc_episode(const Mlp& m0, const Mlp& m1, uint64_t g, uint64_t seed, const float* ext,
                  float* rec_obs, float* rec_logits, int8_t* rec_action, int8_t* rec_seat,
                  int* n_dec) {
    int c0, c1, pub;
    leduc_deal(g, seed, &c0, &c1, &pub);
    Leduc s;
    leduc_init(s, c0, c1, pub);
    int t = 0;
    while (!s.done) {
        float o[17], lg[3];
        leduc_obs(s, o);
        const Mlp& m = (s.actor == 0) ? m0 : m1;
        mlp_logits(m, o, lg);
        uint8_t legal[3];
        leduc_legal(s, legal);
        const float* use = ext ? ext + t * 3 : lg;
        float u = uniform24(draw(g, (uint32_t)t, (uint32_t)s.actor, seed).x[0]);
        int a = sample_masked(use, legal, 3, u);
        if (rec_obs) std::memcpy(rec_obs + t * 17, o, sizeof(o));
        if (rec_logits) std::memcpy(rec_logits + t * 3, lg, sizeof(lg));
        if (rec_action) rec_action[t] = (int8_t)a;
        if (rec_seat) rec_seat[t] = (int8_t)s.actor;
        leduc_apply(s, a);
        ++t;
    }
    if (n_dec) *n_dec = t;
    return s.payoff0;
}

// Exact expected seat-0 payoff of a pair: every ordered deal of the 6 cards
// (6*5*4 = 120, equally likely) times the betting tree, with the policy's
// action probabilities = fp64 softmax of its fp32 logits over legal actions.
// A seat's logits depend only on its observation, so each walk keeps the
// logits of the observations it has met (at most 144 per seat) and looks them
// up instead of running the MLP again: a memo of a pure function, the values
// are the same bits.
struct LogitMemo {
    std::vector<float> obs[2], lg[2];          // per seat: [n][17], [n][3]
    void get(const Mlp& m, int seat, const float* o, float* out) {
        const std::vector<float>& ob = obs[seat];
        for (size_t i = 0; i < ob.size(); i += 17)
            if (std::memcmp(ob.data() + i, o, 17 * sizeof(float)) == 0) {
                std::memcpy(out, lg[seat].data() + i / 17 * 3, 3 * sizeof(float));
                return;
            }
        mlp_logits(m, o, out);
        obs[seat].insert(obs[seat].end(), o, o + 17);
        lg[seat].insert(lg[seat].end(), out, out + 3);
    }
};

double leduc_tree(const Mlp& m0, const Mlp& m1, const Leduc& s, LogitMemo& memo) {
    if (s.done) return (double)s.payoff0;
    float o[17], lg[3];
    leduc_obs(s, o);
    memo.get(s.actor == 0 ? m0 : m1, s.actor, o, lg);
    uint8_t legal[3];
    leduc_legal(s, legal);
    double mx = -1e300;
    for (int a = 0; a < 3; ++a) if (legal[a] && (double)lg[a] > mx) mx = lg[a];
    double z = 0.0, pr[3];
    for (int a = 0; a < 3; ++a) { pr[a] = legal[a] ? std::exp((double)lg[a] - mx) : 0.0; z += pr[a]; }
    double v = 0.0;
    for (int a = 0; a < 3; ++a) {
        if (!legal[a]) continue;
        Leduc n = s;
        leduc_apply(n, a);
        v += (pr[a] / z) * leduc_tree(m0, m1, n, memo);
    }
    return v;
}

double leduc_exact(const Mlp& m0, const Mlp& m1) {
    LogitMemo memo;
    double total = 0.0;
    for (int c0 = 0; c0 < 6; ++c0)
        for (int c1 = 0; c1 < 6; ++c1)
            for (int p = 0; p < 6; ++p) {
                if (c0 == c1 || p == c0 || p == c1) continue;
                Leduc s;
                leduc_init(s, c0, c1, p);
                total += leduc_tree(m0, m1, s, memo) / 120.0;
            }
    return total;
}

// ---------------------------------------------------------------------------
// Cooperative particle spread (App. B.1 semantics; constants of the named
// workloads): N agents and L landmarks; reset: positions and landmarks
// uniform in [-1,1]^2, velocity 0. Step (mass 1, dt 0.1, damping 0.25): v <-
// v*(1-0.25); v <- v + F*dt; p <- p + v*dt; F in {0, +x, -x, +y, -y} of
// magnitude 1 (actions 0..4). Reward after the step, per agent i:
//   r_i = -(sum_l min_a |p_a - l| + #{j != i : |p_i - p_j| < 0.3})
// (radius 0.15 each). Observation of agent i: own velocity, own position,
// landmark positions relative to p_i, other agents' positions relative to p_i
// (ascending j), zero-padded to obs_dim.
// ---------------------------------------------------------------------------
struct Spread {
    int N, L;
    float px[16], py[16], vx[16], vy[16];
    float lx[16], ly[16];
};

void spread_reset(Spread& s, int N, int L, uint64_t g, uint64_t seed) {
    s.N = N; s.L = L;
    for (int i = 0; i < N; ++i) {
        Words w = draw(g, (uint32_t)i, CHANCE, seed);
        s.px[i] = uniform24(w.x[0]) * 2.0f - 1.0f;
        s.py[i] = uniform24(w.x[1]) * 2.0f - 1.0f;
        s.vx[i] = 0.0f; s.vy[i] = 0.0f;
    }
    for (int l = 0; l < L; ++l) {
        Words w = draw(g, 0x80000000u + (uint32_t)l, CHANCE, seed);
        s.lx[l] = uniform24(w.x[0]) * 2.0f - 1.0f;
        s.ly[l] = uniform24(w.x[1]) * 2.0f - 1.0f;
    }
}

void spread_obs(const Spread& s, int i, int obs_dim, float* o) {
    for (int k = 0; k < obs_dim; ++k) o[k] = 0.0f;
    int k = 0;
    o[k++] = s.vx[i]; o[k++] = s.vy[i];
    o[k++] = s.px[i]; o[k++] = s.py[i];
    for (int l = 0; l < s.L; ++l) { o[k++] = s.lx[l] - s.px[i]; o[k++] = s.ly[l] - s.py[i]; }
    for (int j = 0; j < s.N; ++j) {
        if (j == i) continue;
        o[k++] = s.px[j] - s.px[i]; o[k++] = s.py[j] - s.py[i];
    }
}

float dist2d(float ax, float ay, float bx, float by) {
    float dx = ax - bx, dy = ay - by;
    float sq = dx * dx + dy * dy;
    return std::sqrt(sq);
}

// ---------------------------------------------------------------------------
// det_log1pf: log(1 + y) for y in [0, 1] in fp32, every step one correctly
// rounded IEEE operation. Method: log(1 + y) = 2 atanh(z) with z = y / (2 + y)
// in [0, 1/3], and atanh(z) = z (1 + z^2/3 + z^4/5 + ... + z^16/17) (the odd
// power series, truncated after z^17: the next term is below 2^-32 relative),
// in Horner form in w = z^2 with fused multiply-adds.
// ---------------------------------------------------------------------------
float det_log1pf(float y) {
    if (!(y > 0.0f)) return 0.0f;
    const float z = y / (2.0f + y);
    const float w = z * z;
    float p = 0x1.e1e1e2p-5f;         // 1/17
    p = fmaf(p, w, 0x1.111112p-4f);   // 1/15
    p = fmaf(p, w, 0x1.3b13b2p-4f);   // 1/13
    p = fmaf(p, w, 0x1.745d18p-4f);   // 1/11
    p = fmaf(p, w, 0x1.c71c72p-4f);   // 1/9
    p = fmaf(p, w, 0x1.24924ap-3f);   // 1/7
    p = fmaf(p, w, 0x1.99999ap-3f);   // 1/5
    p = fmaf(p, w, 0x1.555556p-2f);   // 1/3
    p = fmaf(p, w, 1.0f);
    return (2.0f * z) * p;
}

// ---------------------------------------------------------------------------
// Contact between two colliding disks (App. B.1 names collisions and
// "obstacles block the way" but gives no force law; this is the soft contact
// model of the particle environments the paper runs, restated as a reading):
// centres a and b, radii summing to dmin, delta = a - b, d = |delta|. The
// penetration is a softplus of the overlap with margin k = 0.001,
//   pen = k * log(1 + exp((dmin - d) / k)),
// and the force on a is F_c * pen * delta / d with F_c = 100 (b gets its
// negative). Evaluated in fp32 in this order: dx, dy, q = dx*dx + dy*dy,
// d = sqrt(q), x = (dmin - d) / k, softplus(x) = max(x, 0) +
// log1p(exp(-|x|)) (det_expf, det_log1pf), pen = k * softplus, c = (F_c * pen)
// / d, force (c*dx, c*dy). No force when d == 0 or pen == 0 (which holds once
// d - dmin >= 87 k, where det_expf gives 0). Returns whether a force acts.
// ---------------------------------------------------------------------------
const float CONTACT_MARGIN = 0.001f;
const float CONTACT_FORCE = 100.0f;

bool contact_force(float ax, float ay, float bx, float by, float dmin, float* fx, float* fy) {
    const float dx = ax - bx, dy = ay - by;
    const float q = dx * dx + dy * dy;
    const float d = std::sqrt(q);
    if (d == 0.0f) return false;
    const float x = (dmin - d) / CONTACT_MARGIN;
    const float ax_ = std::fabs(x);
    const float sp = (x > 0.0f ? x : 0.0f) + det_log1pf(det_expf(-ax_));
    const float pen = CONTACT_MARGIN * sp;
    if (pen == 0.0f) return false;
    const float c = (CONTACT_FORCE * pen) / d;
    *fx = c * dx;
    *fy = c * dy;
    return true;
}

// Adds the contact forces between every pair of the n movable disks (ascending
// pairs a < b; disk i at (px[i], py[i]) with radius rad[i]) to F: a gets +f, b
// gets -f. Then, for every movable disk a (ascending) and every immovable disk
// o (ascending; at (ox[o], oy[o]), radius orad[o]), the force on a. A force is
// added only where one acts, so with no contact F keeps its bits.
void add_contacts(int n, const float* px, const float* py, const float* rad, int m, const float* ox,
                  const float* oy, const float* orad, float* Fx, float* Fy) {
    for (int a = 0; a < n; ++a)
        for (int b = a + 1; b < n; ++b) {
            float fx, fy;
            if (contact_force(px[a], py[a], px[b], py[b], rad[a] + rad[b], &fx, &fy)) {
                Fx[a] = Fx[a] + fx; Fy[a] = Fy[a] + fy;
                Fx[b] = Fx[b] - fx; Fy[b] = Fy[b] - fy;
            }
        }
    for (int a = 0; a < n; ++a)
        for (int o = 0; o < m; ++o) {
            float fx, fy;
            if (contact_force(px[a], py[a], ox[o], oy[o], rad[a] + orad[o], &fx, &fy)) {
                Fx[a] = Fx[a] + fx; Fy[a] = Fy[a] + fy;
            }
        }
}

// Unit action force of the five discrete actions (0 noop, 1 +x, 2 -x, 3 +y, 4 -y).
void action_force(int act, float* fx, float* fy) {
    *fx = 0.0f; *fy = 0.0f;
    switch (act) {
        case 1: *fx = 1.0f; break;
        case 2: *fx = -1.0f; break;
        case 3: *fy = 1.0f; break;
        case 4: *fy = -1.0f; break;
        default: break;
    }
}

// local_ratio < 0: r_i = -(cover + collisions_i) (the workloads' reward);
// otherwise the App. B.1 weighting of the shared and the local term:
// r_i = -((1 - local_ratio) * cover + local_ratio * collisions_i), evaluated
// as written (one rounding per operation, no contraction).
// contact: the agents (radius 0.15) also push each other apart with the soft
// contact forces of add_contacts, computed from the positions before the move
// and added to the action forces (landmarks do not collide).
void spread_step(Spread& s, const int* action, float* reward, float local_ratio, bool contact = false) {
    float Fx[16], Fy[16];
    for (int i = 0; i < s.N; ++i) action_force(action[i], &Fx[i], &Fy[i]);
    if (contact) {
        float rad[16];
        for (int i = 0; i < s.N; ++i) rad[i] = 0.15f;
        add_contacts(s.N, s.px, s.py, rad, 0, nullptr, nullptr, nullptr, Fx, Fy);
    }
    for (int i = 0; i < s.N; ++i) {
        s.vx[i] = s.vx[i] * 0.75f;
        s.vy[i] = s.vy[i] * 0.75f;
        s.vx[i] = s.vx[i] + Fx[i] * 0.1f;
        s.vy[i] = s.vy[i] + Fy[i] * 0.1f;
        s.px[i] = s.px[i] + s.vx[i] * 0.1f;
        s.py[i] = s.py[i] + s.vy[i] * 0.1f;
    }
    float cover = 0.0f;
    for (int l = 0; l < s.L; ++l) {
        float best = dist2d(s.px[0], s.py[0], s.lx[l], s.ly[l]);
        for (int a = 1; a < s.N; ++a) {
            float d = dist2d(s.px[a], s.py[a], s.lx[l], s.ly[l]);
            if (d < best) best = d;
        }
        cover = cover + best;
    }
    for (int i = 0; i < s.N; ++i) {
        int coll = 0;
        for (int j = 0; j < s.N; ++j) {
            if (j == i) continue;
            if (dist2d(s.px[i], s.py[i], s.px[j], s.py[j]) < 0.3f) ++coll;
        }
        if (local_ratio < 0.0f) {
            reward[i] = -(cover + (float)coll);
        } else {
            const float shared = (1.0f - local_ratio) * cover;
            const float local = local_ratio * (float)coll;
            reward[i] = -(shared + local);
        }
    }
}

// ---------------------------------------------------------------------------
// Simple adversary (App. B.1; readings of its description, constants of the
// spread scenario): agent 0 is the adversary, agents 1 and 2 the good agents,
// two landmarks. Reset: agents and landmarks as for spread (same chance
// counters), the target landmark = pick(x of the chance draw with step field
// 0xC0000000, 2). Same dynamics as spread (no contact forces). Rewards after
// the move, with d(.) the distance to the target:
//   good agents: -min(d(p_1), d(p_2)) + d(p_0)      (shared)
//   adversary:   -d(p_0)
// each evaluated as written (one rounding per operation). Observation of agent
// i (14 floats): velocity, position, target - p_i (zeros for the adversary,
// which is not told the target), landmarks - p_i, other agents - p_i
// (ascending j).
// ---------------------------------------------------------------------------
struct Adversary {
    Spread s;
    int target;
};

void adversary_reset(Adversary& a, uint64_t g, uint64_t seed) {
    spread_reset(a.s, 3, 2, g, seed);
    a.target = (int)pick(draw(g, 0xC0000000u, CHANCE, seed).x[0], 2);
}

void adversary_obs(const Adversary& a, int i, float* o) {
    const Spread& s = a.s;
    int k = 0;
    o[k++] = s.vx[i]; o[k++] = s.vy[i];
    o[k++] = s.px[i]; o[k++] = s.py[i];
    if (i == 0) {
        o[k++] = 0.0f; o[k++] = 0.0f;
    } else {
        o[k++] = s.lx[a.target] - s.px[i]; o[k++] = s.ly[a.target] - s.py[i];
    }
    for (int l = 0; l < 2; ++l) { o[k++] = s.lx[l] - s.px[i]; o[k++] = s.ly[l] - s.py[i]; }
    for (int j = 0; j < 3; ++j) {
        if (j == i) continue;
        o[k++] = s.px[j] - s.px[i]; o[k++] = s.py[j] - s.py[i];
    }
}

void adversary_step(Adversary& a, const int* action, float* reward) {
    Spread& s = a.s;
    for (int i = 0; i < 3; ++i) {
        float fx = 0.0f, fy = 0.0f;
        switch (action[i]) {
            case 1: fx = 1.0f; break;
            case 2: fx = -1.0f; break;
            case 3: fy = 1.0f; break;
            case 4: fy = -1.0f; break;
            default: break;
        }
        s.vx[i] = s.vx[i] * 0.75f;
        s.vy[i] = s.vy[i] * 0.75f;
        s.vx[i] = s.vx[i] + fx * 0.1f;
        s.vy[i] = s.vy[i] + fy * 0.1f;
        s.px[i] = s.px[i] + s.vx[i] * 0.1f;
        s.py[i] = s.py[i] + s.vy[i] * 0.1f;
    }
    const float tx = s.lx[a.target], ty = s.ly[a.target];
    const float d_adv = dist2d(s.px[0], s.py[0], tx, ty);
    const float d1 = dist2d(s.px[1], s.py[1], tx, ty);
    const float d2 = dist2d(s.px[2], s.py[2], tx, ty);
    const float d_good = d1 < d2 ? d1 : d2;
    reward[0] = -d_adv;
    reward[1] = -d_good + d_adv;
    reward[2] = reward[1];
}

// ---------------------------------------------------------------------------
// Simple speaker listener (App. B.1; readings of its description and of the
// simple reference scenario it is said to resemble, constants of the spread
// scenario): agent 0 is the speaker, which does not move and whose action
// 0..2 is the message it sends (actions 3 and 4 are not legal for it); agent 1
// the listener, which moves with the spread dynamics and cannot speak; three
// landmarks, one of them the target. Reset: agents and landmarks as for spread
// (same chance counters), the target = pick(x of the chance draw with step
// field 0xC0000000, 3), no message yet. The listener observes the message the
// speaker sent at the previous step. Reward after the move, shared by both
// agents: -d(p_1, target). Observations (11 floats): speaker - one-hot of the
// target, zeros; listener - velocity, landmarks - p_1 (ascending), one-hot of
// the last message (zeros before the first).
// ---------------------------------------------------------------------------
struct SpeakerListener {
    Spread s;
    int target;
    int msg;            // -1: none yet
};

void sl_reset(SpeakerListener& a, uint64_t g, uint64_t seed) {
    spread_reset(a.s, 2, 3, g, seed);
    a.target = (int)pick(draw(g, 0xC0000000u, CHANCE, seed).x[0], 3);
    a.msg = -1;
}

void sl_obs(const SpeakerListener& a, int i, float* o) {
    for (int k = 0; k < 11; ++k) o[k] = 0.0f;
    const Spread& s = a.s;
    if (i == 0) {
        o[a.target] = 1.0f;
        return;
    }
    int k = 0;
    o[k++] = s.vx[1]; o[k++] = s.vy[1];
    for (int l = 0; l < 3; ++l) { o[k++] = s.lx[l] - s.px[1]; o[k++] = s.ly[l] - s.py[1]; }
    if (a.msg >= 0) o[k + a.msg] = 1.0f;
}

void sl_step(SpeakerListener& a, const int* action, float* reward) {
    Spread& s = a.s;
    a.msg = action[0];
    float fx = 0.0f, fy = 0.0f;
    switch (action[1]) {
        case 1: fx = 1.0f; break;
        case 2: fx = -1.0f; break;
        case 3: fy = 1.0f; break;
        case 4: fy = -1.0f; break;
        default: break;
    }
    s.vx[1] = s.vx[1] * 0.75f;
    s.vy[1] = s.vy[1] * 0.75f;
    s.vx[1] = s.vx[1] + fx * 0.1f;
    s.vy[1] = s.vy[1] + fy * 0.1f;
    s.px[1] = s.px[1] + s.vx[1] * 0.1f;
    s.py[1] = s.py[1] + s.vy[1] * 0.1f;
    const float d = dist2d(s.px[1], s.py[1], s.lx[a.target], s.ly[a.target]);
    reward[0] = -d;
    reward[1] = -d;
}

// ---------------------------------------------------------------------------
// Simple push (App. B.1; readings of its description, constants of the spread
// scenario): agent 0 is the adversary, agent 1 the good agent, one landmark.
// Reset as spread (same chance counters, N = 2, L = 1). Both agents are disks
// of radius 0.15 that push each other with the soft contact forces (the
// landmark does not collide); unit action forces, mass 1, dt 0.1, damping
// 0.25. Rewards after the move, with d_i = |p_i - landmark|:
//   good agent r_1 = -d_1;   adversary r_0 = d_1 - d_0
// (close to the landmark itself, and the good agent far from it: the
// difference of the distances). Observation of agent i (8 floats): velocity,
// position, landmark - p_i, the other agent - p_i.
// ---------------------------------------------------------------------------
struct Push {
    Spread s;
};

void push_reset(Push& a, uint64_t g, uint64_t seed) { spread_reset(a.s, 2, 1, g, seed); }

void push_obs(const Push& a, int i, float* o) {
    const Spread& s = a.s;
    const int j = 1 - i;
    o[0] = s.vx[i]; o[1] = s.vy[i];
    o[2] = s.px[i]; o[3] = s.py[i];
    o[4] = s.lx[0] - s.px[i]; o[5] = s.ly[0] - s.py[i];
    o[6] = s.px[j] - s.px[i]; o[7] = s.py[j] - s.py[i];
}

void push_step(Push& a, const int* action, float* reward) {
    Spread& s = a.s;
    float Fx[2], Fy[2];
    for (int i = 0; i < 2; ++i) action_force(action[i], &Fx[i], &Fy[i]);
    const float rad[2] = {0.15f, 0.15f};
    add_contacts(2, s.px, s.py, rad, 0, nullptr, nullptr, nullptr, Fx, Fy);
    for (int i = 0; i < 2; ++i) {
        s.vx[i] = s.vx[i] * 0.75f;
        s.vy[i] = s.vy[i] * 0.75f;
        s.vx[i] = s.vx[i] + Fx[i] * 0.1f;
        s.vy[i] = s.vy[i] + Fy[i] * 0.1f;
        s.px[i] = s.px[i] + s.vx[i] * 0.1f;
        s.py[i] = s.py[i] + s.vy[i] * 0.1f;
    }
    const float d0 = dist2d(s.px[0], s.py[0], s.lx[0], s.ly[0]);
    const float d1 = dist2d(s.px[1], s.py[1], s.lx[0], s.ly[0]);
    reward[0] = d1 - d0;
    reward[1] = -d1;
}

// ---------------------------------------------------------------------------
// Simple tag (App. B.1; readings of its description: "the good agent is
// faster", "-10 for each collision" / "+10 for each collision", "obstacles
// block the way"; sizes, accelerations and speed limits as stated readings):
// agents 0..2 are the adversaries (radius 0.075, action force 3, speed limit
// 1.0), agent 3 the good agent (radius 0.05, action force 4, speed limit 1.3),
// two obstacles (radius 0.2, immovable). Reset as spread (same chance
// counters, N = 4, the obstacles in the landmark slots L = 2). Every pair of
// agents and every (agent, obstacle) pair collides with the soft contact
// forces, from the positions before the move. Per agent (ascending): v <- v *
// 0.75; v <- v + F * 0.1 (mass 1); if |v| > limit, v <- (v / |v|) * limit per
// component; p <- p + v * 0.1. After the move adversary i hits the good agent
// when |p_i - p_3| < 0.075 + 0.05; with h the number of hits, r_3 = -10 h and
// every adversary gets r_i = 10 h. Observation of agent i (16 floats):
// velocity, position, obstacles - p_i, the other agents - p_i (ascending),
// then the good agent's velocity for an adversary (zeros for the good agent).
// ---------------------------------------------------------------------------
struct Tag {
    Spread s;
};

const float TAG_RAD[4] = {0.075f, 0.075f, 0.075f, 0.05f};
const float TAG_ACCEL[4] = {3.0f, 3.0f, 3.0f, 4.0f};
const float TAG_VMAX[4] = {1.0f, 1.0f, 1.0f, 1.3f};
const float TAG_OBST_RAD[2] = {0.2f, 0.2f};

void tag_reset(Tag& a, uint64_t g, uint64_t seed) { spread_reset(a.s, 4, 2, g, seed); }

void tag_obs(const Tag& a, int i, float* o) {
    const Spread& s = a.s;
    int k = 0;
    o[k++] = s.vx[i]; o[k++] = s.vy[i];
    o[k++] = s.px[i]; o[k++] = s.py[i];
    for (int l = 0; l < 2; ++l) { o[k++] = s.lx[l] - s.px[i]; o[k++] = s.ly[l] - s.py[i]; }
    for (int j = 0; j < 4; ++j) {
        if (j == i) continue;
        o[k++] = s.px[j] - s.px[i]; o[k++] = s.py[j] - s.py[i];
    }
    if (i < 3) { o[k++] = s.vx[3]; o[k++] = s.vy[3]; }
    else { o[k++] = 0.0f; o[k++] = 0.0f; }
}

void tag_step(Tag& a, const int* action, float* reward) {
    Spread& s = a.s;
    float Fx[4], Fy[4];
    for (int i = 0; i < 4; ++i) {
        float ux, uy;
        action_force(action[i], &ux, &uy);
        Fx[i] = TAG_ACCEL[i] * ux;
        Fy[i] = TAG_ACCEL[i] * uy;
    }
    add_contacts(4, s.px, s.py, TAG_RAD, 2, s.lx, s.ly, TAG_OBST_RAD, Fx, Fy);
    for (int i = 0; i < 4; ++i) {
        s.vx[i] = s.vx[i] * 0.75f;
        s.vy[i] = s.vy[i] * 0.75f;
        s.vx[i] = s.vx[i] + Fx[i] * 0.1f;
        s.vy[i] = s.vy[i] + Fy[i] * 0.1f;
        const float speed = std::sqrt(s.vx[i] * s.vx[i] + s.vy[i] * s.vy[i]);
        if (speed > TAG_VMAX[i]) {
            s.vx[i] = (s.vx[i] / speed) * TAG_VMAX[i];
            s.vy[i] = (s.vy[i] / speed) * TAG_VMAX[i];
        }
        s.px[i] = s.px[i] + s.vx[i] * 0.1f;
        s.py[i] = s.py[i] + s.vy[i] * 0.1f;
    }
    int hits = 0;
    for (int i = 0; i < 3; ++i)
        if (dist2d(s.px[i], s.py[i], s.px[3], s.py[3]) < TAG_RAD[i] + TAG_RAD[3]) ++hits;
    for (int i = 0; i < 3; ++i) reward[i] = 10.0f * (float)hits;
    reward[3] = -10.0f * (float)hits;
}

// ---------------------------------------------------------------------------
// Simple reference (App. B.1; readings of its description and of the speaker
// listener it is said to resemble): two agents, three landmarks; each agent has
// a goal landmark that only the other agent is told; both are speakers and
// listeners. An action is a move and a message at once: a = 5 * message +
// move (move 0..4 as in spread, message 0..2 naming a landmark), 15 actions.
// Reset as spread (N = 2, L = 3, same chance counters); agent i's goal =
// pick(x of the chance draw with step field 0xC0000000 + i, 3); no message yet.
// Step: the spread dynamics for both agents (no contact), then each agent's
// message is stored, seen by the other agent from the next step on. Rewards
// after the move, d_i = |p_i - goal landmark of i|, rho = local_ratio (0.5
// unless given): r_i = -((1 - rho) * ((d_0 + d_1) * 0.5) + rho * d_i) ("locally
// ... their distance to their target landmark; globally ... the average
// distance"), each operation rounded in fp32 in this order. Observation of
// agent i (14 floats): velocity, the three landmarks - p_i, the other agent's
// goal as a one-hot, the other agent's last message as a one-hot (zeros before
// the first).
// ---------------------------------------------------------------------------
struct Reference {
    Spread s;
    int goal[2];
    int msg[2];          // -1: none yet
    float rho;
};

void ref_reset(Reference& a, uint64_t g, uint64_t seed) {
    spread_reset(a.s, 2, 3, g, seed);
    for (int i = 0; i < 2; ++i) {
        a.goal[i] = (int)pick(draw(g, 0xC0000000u + (uint32_t)i, CHANCE, seed).x[0], 3);
        a.msg[i] = -1;
    }
}

void ref_obs(const Reference& a, int i, float* o) {
    const Spread& s = a.s;
    const int j = 1 - i;
    for (int k = 0; k < 14; ++k) o[k] = 0.0f;
    o[0] = s.vx[i]; o[1] = s.vy[i];
    for (int l = 0; l < 3; ++l) { o[2 + 2 * l] = s.lx[l] - s.px[i]; o[3 + 2 * l] = s.ly[l] - s.py[i]; }
    o[8 + a.goal[j]] = 1.0f;
    if (a.msg[j] >= 0) o[11 + a.msg[j]] = 1.0f;
}

void ref_step(Reference& a, const int* action, float* reward) {
    Spread& s = a.s;
    for (int i = 0; i < 2; ++i) {
        float fx, fy;
        action_force(action[i] % 5, &fx, &fy);
        s.vx[i] = s.vx[i] * 0.75f;
        s.vy[i] = s.vy[i] * 0.75f;
        s.vx[i] = s.vx[i] + fx * 0.1f;
        s.vy[i] = s.vy[i] + fy * 0.1f;
        s.px[i] = s.px[i] + s.vx[i] * 0.1f;
        s.py[i] = s.py[i] + s.vy[i] * 0.1f;
    }
    for (int i = 0; i < 2; ++i) a.msg[i] = action[i] / 5;
    float d[2];
    for (int i = 0; i < 2; ++i) d[i] = dist2d(s.px[i], s.py[i], s.lx[a.goal[i]], s.ly[a.goal[i]]);
    const float mean = (d[0] + d[1]) * 0.5f;
    for (int i = 0; i < 2; ++i) {
        const float shared = (1.0f - a.rho) * mean;
        const float local = a.rho * d[i];
        reward[i] = -(shared + local);
    }
}

// One rollout driver for the fixed-size scenarios (push, tag, reference): Env
// supplies N, IN, A, reset, obs and step; all actions legal.
struct PushEnvDef {
    using S = Push;
    static const int N = 2, IN = 8, A = 5;
    static void reset(S& a, uint64_t g, uint64_t seed) { push_reset(a, g, seed); }
    static void obs(const S& a, int i, float* o) { push_obs(a, i, o); }
    static void step(S& a, const int* act, float* r) { push_step(a, act, r); }
};
struct TagEnvDef {
    using S = Tag;
    static const int N = 4, IN = 16, A = 5;
    static void reset(S& a, uint64_t g, uint64_t seed) { tag_reset(a, g, seed); }
    static void obs(const S& a, int i, float* o) { tag_obs(a, i, o); }
    static void step(S& a, const int* act, float* r) { tag_step(a, act, r); }
};
struct RefEnvDef {
    using S = Reference;
    static const int N = 2, IN = 14, A = 15;
    static float rho;
    static void reset(S& a, uint64_t g, uint64_t seed) { ref_reset(a, g, seed); a.rho = rho; }
    static void obs(const S& a, int i, float* o) { ref_obs(a, i, o); }
    static void step(S& a, const int* act, float* r) { ref_step(a, act, r); }
};
float RefEnvDef::rho = 0.5f;

template <class Env>
void scenario_rollout(const float* const* params, int h1, int h2, int bf16, int T, int64_t n_envs,
                      int64_t env_lo, int64_t env_hi, const int32_t* pairs, int32_t n_pairs,
                      int64_t n_episodes, uint64_t seed, const float* ext_logits, float* obs,
                      int8_t* action, float* reward, float* logits, int n_threads) {
    const int N = Env::N, in = Env::IN, A = Env::A;
    int64_t per = n_envs / n_pairs;
    int64_t W = env_hi - env_lo;
    parallel_for(W * n_episodes, n_threads, [&](int64_t job) {
        int64_t ep = job / W, e = env_lo + job % W;
        int64_t row = e / per;
        typename Env::S st;
        uint64_t g = (uint64_t)ep * (uint64_t)n_envs + (uint64_t)e;
        Env::reset(st, g, seed);
        for (int t = 0; t < T; ++t) {
            int act[Env::N];
            for (int i = 0; i < N; ++i) {
                int64_t idx = ((ep * T + t) * W + (e - env_lo)) * N + i;
                float o[Env::IN], lg[16];
                Env::obs(st, i, o);
                Mlp m{params[pairs[row * N + i]], in, h1, h2, A, bf16};
                mlp_logits(m, o, lg);
                uint8_t legal[16];
                for (int q = 0; q < 16; ++q) legal[q] = 1;
                float u = uniform24(draw(g, (uint32_t)t, (uint32_t)i, seed).x[0]);
                act[i] = sample_masked(ext_logits ? ext_logits + idx * A : lg, legal, A, u);
                if (obs) std::memcpy(obs + idx * in, o, sizeof(float) * in);
                if (logits) std::memcpy(logits + idx * A, lg, sizeof(float) * A);
                if (action) action[idx] = (int8_t)act[i];
            }
            float r[Env::N];
            Env::step(st, act, r);
            if (reward)
                for (int i = 0; i < N; ++i) reward[((ep * T + t) * W + (e - env_lo)) * N + i] = r[i];
        }
    });
}

}  // namespace

// ===========================================================================
// C entry points (loaded by the tests and the benchmark's CPU-baseline leg).
// ===========================================================================
extern "C" {

void orc_philox(const uint32_t* ctr, uint64_t seed, uint32_t* out, int64_t n) {
    for (int64_t i = 0; i < n; ++i) {
        Words w = philox4x32_10(ctr[4 * i], ctr[4 * i + 1], ctr[4 * i + 2], ctr[4 * i + 3], seed);
        for (int k = 0; k < 4; ++k) out[4 * i + k] = w.x[k];
    }
}

void orc_det_expf(const float* x, float* y, int64_t n) {
    for (int64_t i = 0; i < n; ++i) y[i] = det_expf(x[i]);
}

void orc_det_log1pf(const float* x, float* y, int64_t n) {
    for (int64_t i = 0; i < n; ++i) y[i] = det_log1pf(x[i]);
}

// Contact force on disk a from disk b (radii summing to dmin): out[0..1] the
// force, out[2] = 1 when one acts (else 0 and a zero force).
void orc_contact_force(float ax, float ay, float bx, float by, float dmin, float* out) {
    float fx = 0.0f, fy = 0.0f;
    const bool on = contact_force(ax, ay, bx, by, dmin, &fx, &fy);
    out[0] = fx; out[1] = fy; out[2] = on ? 1.0f : 0.0f;
}

void orc_sample(const float* logits, const uint8_t* legal, const float* u, int A, int32_t* out, int64_t n) {
    for (int64_t i = 0; i < n; ++i) out[i] = sample_masked(logits + i * A, legal + i * A, A, u[i]);
}

float orc_bf16_round(float x) { return bf16_round(x); }

void orc_mlp_forward(const float* params, int in, int h1, int h2, int out, int bf16,
                     const float* x, int64_t n, float* logits) {
    Mlp m{params, in, h1, h2, out, bf16};
    for (int64_t r = 0; r < n; ++r) mlp_logits(m, x + r * in, logits + r * out);
}

// ---- Kuhn ----
double orc_kuhn_exact(const float* pol0, const float* pol1) { return kuhn_exact(pol0, pol1); }

// pol: [n_pol][6]; pairs: [n_pairs][2]; out: [n_pairs][4] (mean, SE, sum, sumsq).
// trace (optional): per pair, per episode < n_trace: card0, card1, n_dec,
// action[3] (-1 padded), payoff0  -> int32[n_pairs][n_trace][8].
void orc_kuhn_eval(const float* pol, const int32_t* pairs, int32_t n_pairs, int64_t n_episodes,
                   uint64_t seed, double* out, int32_t* trace, int64_t n_trace, int n_threads) {
    parallel_for(n_pairs, n_threads, [&](int64_t p) {
        const float* p0 = pol + 6 * (int64_t)pairs[2 * p];
        const float* p1 = pol + 6 * (int64_t)pairs[2 * p + 1];
        int64_t s1 = 0, s2 = 0;
        for (int64_t e = 0; e < n_episodes; ++e) {
            uint64_t g = (uint64_t)p * (uint64_t)n_episodes + (uint64_t)e;
            KuhnTrace tr;
            int r = kuhn_episode(p0, p1, g, seed, &tr);
            s1 += r; s2 += (int64_t)r * r;
            if (trace && e < n_trace) {
                int32_t* t = trace + (p * n_trace + e) * 8;
                t[0] = tr.card0; t[1] = tr.card1; t[2] = tr.n_dec;
                for (int k = 0; k < 3; ++k) t[3 + k] = k < tr.n_dec ? tr.action[k] : -1;
                t[6] = tr.payoff0; t[7] = 0;
            }
        }
        finish_entry(s1, s2, n_episodes, out + 4 * p);
    });
}

// Plays n hands with global episode ids g0 .. g0 + n - 1 (Sec. 4.2's simulations
// indexed as in orc_kuhn_eval), for checking records of hands whose id is
// too far into a long evaluation for the whole evaluation to be replayed.
// trace [n][8] as in orc_kuhn_eval.
void orc_kuhn_hands(const float* pol0, const float* pol1, uint64_t g0, int64_t n, uint64_t seed,
                    int32_t* trace) {
    for (int64_t e = 0; e < n; ++e) {
        KuhnTrace tr;
        kuhn_episode(pol0, pol1, g0 + (uint64_t)e, seed, &tr);
        int32_t* t = trace + e * 8;
        t[0] = tr.card0; t[1] = tr.card1; t[2] = tr.n_dec;
        for (int k = 0; k < 3; ++k) t[3 + k] = k < tr.n_dec ? tr.action[k] : -1;
        t[6] = tr.payoff0; t[7] = 0;
    }
}

// ---- Leduc ----
void orc_leduc_deal(uint64_t g, uint64_t seed, int32_t* cards3) {
    int a, b, c;
    leduc_deal(g, seed, &a, &b, &c);
    cards3[0] = a; cards3[1] = b; cards3[2] = c;
}

// Plays a fixed action sequence from a fixed deal. Returns the number of
// actions consumed before the hand ended, or -1 at the first illegal action.
// Outputs: payoff0, contributions, and per decision the acting seat, the
// 17-float observation and the legal mask.
int orc_leduc_play(int c0, int c1, int pub, const int32_t* actions, int n, int32_t* payoff0,
                   int32_t* contrib2, int32_t* seats, float* obs, uint8_t* legal, int32_t* done) {
    Leduc s;
    leduc_init(s, c0, c1, pub);
    int t = 0;
    for (; t < n && !s.done; ++t) {
        if (seats) seats[t] = s.actor;
        if (obs) leduc_obs(s, obs + 17 * t);
        if (legal) leduc_legal(s, legal + 3 * t);
        if (leduc_apply(s, actions[t]) != 0) return -1;
    }
    if (payoff0) *payoff0 = s.payoff0;
    if (contrib2) { contrib2[0] = s.contrib[0]; contrib2[1] = s.contrib[1]; }
    if (done) *done = s.done;
    return t;
}

double orc_leduc_exact(const float* params0, const float* params1, int in, int h1, int h2, int out,
                       int bf16) {
    Mlp m0{params0, in, h1, h2, out, bf16}, m1{params1, in, h1, h2, out, bf16};
    return leduc_exact(m0, m1);
}

// params: [n_pol] pointers to the plain layout; pairs [n_pairs][2].
// Simulates hands e in [0, n_sim) of every pair, with global episode ids
// g = pair * n_episodes + e; out [n_pairs][4] summarises those n_sim hands. Optional per-episode records for episodes e < n_rec of every
// pair: obs [n_pairs][n_rec][8][17], logits [..][8][3], action/seat int8
// [..][8] (-1 after the end), payoff int32 [n_pairs][n_rec], ndec int32.
// ext_logits (optional, [n_pairs][n_rec][8][3]) drives the draws of those
// episodes instead of the oracle's own logits.
void orc_leduc_eval(const float* const* params, int in, int h1, int h2, int out, int bf16,
                    const int32_t* pairs, int32_t n_pairs, int64_t n_episodes, int64_t n_sim,
                    uint64_t seed, double* res, int64_t n_rec, const float* ext_logits, float* rec_obs,
                    float* rec_logits, int8_t* rec_action, int8_t* rec_seat, int32_t* rec_payoff,
                    int32_t* rec_ndec, int64_t* dec_per_pair, int n_threads) {
    parallel_for(n_pairs, n_threads, [&](int64_t p) {
        Mlp m0{params[pairs[2 * p]], in, h1, h2, out, bf16};
        Mlp m1{params[pairs[2 * p + 1]], in, h1, h2, out, bf16};
        int64_t s1 = 0, s2 = 0, nd = 0;
        for (int64_t e = 0; e < n_sim; ++e) {
            uint64_t g = (uint64_t)p * (uint64_t)n_episodes + (uint64_t)e;
            bool rec = e < n_rec;
            int64_t base = p * n_rec + e;
            int n_dec = 0;
            int r;
            if (rec) {
                int8_t* ra = rec_action ? rec_action + base * LEDUC_MAX_DEC : nullptr;
                int8_t* rs = rec_seat ? rec_seat + base * LEDUC_MAX_DEC : nullptr;
                if (ra) for (int k = 0; k < LEDUC_MAX_DEC; ++k) ra[k] = -1;
                if (rs) for (int k = 0; k < LEDUC_MAX_DEC; ++k) rs[k] = -1;
                r = leduc_episode(m0, m1, g, seed,
                                  ext_logits ? ext_logits + base * LEDUC_MAX_DEC * 3 : nullptr,
                                  rec_obs ? rec_obs + base * LEDUC_MAX_DEC * 17 : nullptr,
                                  rec_logits ? rec_logits + base * LEDUC_MAX_DEC * 3 : nullptr,
                                  ra, rs, &n_dec);
                if (rec_payoff) rec_payoff[base] = r;
                if (rec_ndec) rec_ndec[base] = n_dec;
            } else {
                r = leduc_episode(m0, m1, g, seed, nullptr, nullptr, nullptr, nullptr, nullptr, &n_dec);
            }
            s1 += r; s2 += (int64_t)r * r;
            nd += n_dec;
        }
        finish_entry(s1, s2, n_sim, res + 4 * p);
        if (dec_per_pair) dec_per_pair[p] = nd;
    });
}

// ---- Spread ----
// One transition from a given state (for hand-worked checks). state: px,py,vx,vy
// for N agents then lx,ly for L landmarks (packed [4N + 2L]); updated in place.
void orc_spread_step(int N, int L, float* state, const int32_t* action, float* reward,
                     float local_ratio, int contact) {
    Spread s;
    s.N = N; s.L = L;
    for (int i = 0; i < N; ++i) {
        s.px[i] = state[4 * i]; s.py[i] = state[4 * i + 1];
        s.vx[i] = state[4 * i + 2]; s.vy[i] = state[4 * i + 3];
    }
    for (int l = 0; l < L; ++l) { s.lx[l] = state[4 * N + 2 * l]; s.ly[l] = state[4 * N + 2 * l + 1]; }
    spread_step(s, action, reward, local_ratio, contact != 0);
    for (int i = 0; i < N; ++i) {
        state[4 * i] = s.px[i]; state[4 * i + 1] = s.py[i];
        state[4 * i + 2] = s.vx[i]; state[4 * i + 3] = s.vy[i];
    }
}

void orc_spread_obs(int N, int L, const float* state, int obs_dim, float* obs /*[N][obs_dim]*/) {
    Spread s;
    s.N = N; s.L = L;
    for (int i = 0; i < N; ++i) {
        s.px[i] = state[4 * i]; s.py[i] = state[4 * i + 1];
        s.vx[i] = state[4 * i + 2]; s.vy[i] = state[4 * i + 3];
    }
    for (int l = 0; l < L; ++l) { s.lx[l] = state[4 * N + 2 * l]; s.ly[l] = state[4 * N + 2 * l + 1]; }
    for (int i = 0; i < N; ++i) spread_obs(s, i, obs_dim, obs + i * obs_dim);
}

void orc_spread_reset(int N, int L, uint64_t g, uint64_t seed, float* state) {
    Spread s;
    spread_reset(s, N, L, g, seed);
    for (int i = 0; i < N; ++i) {
        state[4 * i] = s.px[i]; state[4 * i + 1] = s.py[i];
        state[4 * i + 2] = s.vx[i]; state[4 * i + 3] = s.vy[i];
    }
    for (int l = 0; l < L; ++l) { state[4 * N + 2 * l] = s.lx[l]; state[4 * N + 2 * l + 1] = s.ly[l]; }
}

// Rollout of envs [env_lo, env_hi) for episodes [0, n_episodes):
// env e belongs to combination e / (n_envs / n_pairs); its agent i acts with
// policy pairs[row][i]. g = episode * n_envs + env. Outputs over the slice,
// indexed [ep][t][env - env_lo][agent]: obs [..][obs_dim], action int8,
// reward f32, logits [..][A] (the oracle's own). ext_logits (optional, same
// indexing as logits) drives the draws instead of the oracle's own.
void orc_spread_rollout(const float* const* params, int in, int h1, int h2, int A, int bf16,
                        int N, int L, int T, int64_t n_envs, int64_t env_lo, int64_t env_hi,
                        const int32_t* pairs, int32_t n_pairs, int64_t n_episodes, uint64_t seed,
                        const float* ext_logits, float* obs, int8_t* action, float* reward,
                        float* logits, int n_threads, float local_ratio, int contact) {
    int64_t per = n_envs / n_pairs;
    int64_t W = env_hi - env_lo;
    parallel_for(W * n_episodes, n_threads, [&](int64_t job) {
        int64_t ep = job / W, e = env_lo + job % W;
        int64_t row = e / per;
        Spread s;
        uint64_t g = (uint64_t)ep * (uint64_t)n_envs + (uint64_t)e;
        spread_reset(s, N, L, g, seed);
        for (int t = 0; t < T; ++t) {
            int act[16];
            for (int i = 0; i < N; ++i) {
                int64_t idx = ((ep * T + t) * W + (e - env_lo)) * N + i;
                float o[64], lg[8];
                spread_obs(s, i, in, o);
                Mlp m{params[pairs[row * N + i]], in, h1, h2, A, bf16};
                mlp_logits(m, o, lg);
                uint8_t legal[8] = {1, 1, 1, 1, 1, 1, 1, 1};
                float u = uniform24(draw(g, (uint32_t)t, (uint32_t)i, seed).x[0]);
                act[i] = sample_masked(ext_logits ? ext_logits + idx * A : lg, legal, A, u);
                if (obs) std::memcpy(obs + idx * in, o, sizeof(float) * in);
                if (logits) std::memcpy(logits + idx * A, lg, sizeof(float) * A);
                if (action) action[idx] = (int8_t)act[i];
            }
            float r[16];
            spread_step(s, act, r, local_ratio, contact != 0);
            if (reward)
                for (int i = 0; i < N; ++i) reward[((ep * T + t) * W + (e - env_lo)) * N + i] = r[i];
        }
    });
}

// ---- Simple adversary ----
// state: px,py,vx,vy of the 3 agents, lx,ly of the 2 landmarks, then the
// target index as a float ([4*3 + 2*2 + 1] = 17 floats).
static void adv_load(const float* state, Adversary& a) {
    a.s.N = 3; a.s.L = 2;
    for (int i = 0; i < 3; ++i) {
        a.s.px[i] = state[4 * i]; a.s.py[i] = state[4 * i + 1];
        a.s.vx[i] = state[4 * i + 2]; a.s.vy[i] = state[4 * i + 3];
    }
    for (int l = 0; l < 2; ++l) { a.s.lx[l] = state[12 + 2 * l]; a.s.ly[l] = state[12 + 2 * l + 1]; }
    a.target = (int)state[16];
}
static void adv_store(const Adversary& a, float* state) {
    for (int i = 0; i < 3; ++i) {
        state[4 * i] = a.s.px[i]; state[4 * i + 1] = a.s.py[i];
        state[4 * i + 2] = a.s.vx[i]; state[4 * i + 3] = a.s.vy[i];
    }
    for (int l = 0; l < 2; ++l) { state[12 + 2 * l] = a.s.lx[l]; state[12 + 2 * l + 1] = a.s.ly[l]; }
    state[16] = (float)a.target;
}

void orc_adversary_reset(uint64_t g, uint64_t seed, float* state) {
    Adversary a;
    adversary_reset(a, g, seed);
    adv_store(a, state);
}

void orc_adversary_step(float* state, const int32_t* action, float* reward) {
    Adversary a;
    adv_load(state, a);
    adversary_step(a, action, reward);
    adv_store(a, state);
}

void orc_adversary_obs(const float* state, float* obs /*[3][14]*/) {
    Adversary a;
    adv_load(state, a);
    for (int i = 0; i < 3; ++i) adversary_obs(a, i, obs + i * 14);
}

// Rollout as orc_spread_rollout, for the simple adversary (N = 3, obs 14).
void orc_adversary_rollout(const float* const* params, int h1, int h2, int bf16, int T,
                           int64_t n_envs, int64_t env_lo, int64_t env_hi, const int32_t* pairs,
                           int32_t n_pairs, int64_t n_episodes, uint64_t seed,
                           const float* ext_logits, float* obs, int8_t* action, float* reward,
                           float* logits, int n_threads) {
    const int N = 3, in = 14, A = 5;
    int64_t per = n_envs / n_pairs;
    int64_t W = env_hi - env_lo;
    parallel_for(W * n_episodes, n_threads, [&](int64_t job) {
        int64_t ep = job / W, e = env_lo + job % W;
        int64_t row = e / per;
        Adversary adv;
        uint64_t g = (uint64_t)ep * (uint64_t)n_envs + (uint64_t)e;
        adversary_reset(adv, g, seed);
        for (int t = 0; t < T; ++t) {
            int act[3];
            for (int i = 0; i < N; ++i) {
                int64_t idx = ((ep * T + t) * W + (e - env_lo)) * N + i;
                float o[14], lg[8];
                adversary_obs(adv, i, o);
                Mlp m{params[pairs[row * N + i]], in, h1, h2, A, bf16};
                mlp_logits(m, o, lg);
                uint8_t legal[8] = {1, 1, 1, 1, 1, 1, 1, 1};
                float u = uniform24(draw(g, (uint32_t)t, (uint32_t)i, seed).x[0]);
                act[i] = sample_masked(ext_logits ? ext_logits + idx * A : lg, legal, A, u);
                if (obs) std::memcpy(obs + idx * in, o, sizeof(float) * in);
                if (logits) std::memcpy(logits + idx * A, lg, sizeof(float) * A);
                if (action) action[idx] = (int8_t)act[i];
            }
            float r[3];
            adversary_step(adv, act, r);
            if (reward)
                for (int i = 0; i < N; ++i) reward[((ep * T + t) * W + (e - env_lo)) * N + i] = r[i];
        }
    });
}

// ---- Simple speaker listener ----
// state: px,py,vx,vy of the 2 agents, lx,ly of the 3 landmarks, the target
// index and the last message (-1: none) as floats ([4*2 + 2*3 + 2] = 16).
static void sl_load(const float* state, SpeakerListener& a) {
    a.s.N = 2; a.s.L = 3;
    for (int i = 0; i < 2; ++i) {
        a.s.px[i] = state[4 * i]; a.s.py[i] = state[4 * i + 1];
        a.s.vx[i] = state[4 * i + 2]; a.s.vy[i] = state[4 * i + 3];
    }
    for (int l = 0; l < 3; ++l) { a.s.lx[l] = state[8 + 2 * l]; a.s.ly[l] = state[8 + 2 * l + 1]; }
    a.target = (int)state[14];
    a.msg = (int)state[15];
}
static void sl_store(const SpeakerListener& a, float* state) {
    for (int i = 0; i < 2; ++i) {
        state[4 * i] = a.s.px[i]; state[4 * i + 1] = a.s.py[i];
        state[4 * i + 2] = a.s.vx[i]; state[4 * i + 3] = a.s.vy[i];
    }
    for (int l = 0; l < 3; ++l) { state[8 + 2 * l] = a.s.lx[l]; state[8 + 2 * l + 1] = a.s.ly[l]; }
    state[14] = (float)a.target;
    state[15] = (float)a.msg;
}

void orc_sl_reset(uint64_t g, uint64_t seed, float* state) {
    SpeakerListener a;
    sl_reset(a, g, seed);
    sl_store(a, state);
}

void orc_sl_step(float* state, const int32_t* action, float* reward) {
    SpeakerListener a;
    sl_load(state, a);
    sl_step(a, action, reward);
    sl_store(a, state);
}

void orc_sl_obs(const float* state, float* obs /*[2][11]*/) {
    SpeakerListener a;
    sl_load(state, a);
    for (int i = 0; i < 2; ++i) sl_obs(a, i, obs + i * 11);
}

// Rollout as orc_spread_rollout, for the simple speaker listener (N = 2, obs
// 11, 5 actions of which the speaker may take 0..2).
void orc_sl_rollout(const float* const* params, int h1, int h2, int bf16, int T, int64_t n_envs,
                    int64_t env_lo, int64_t env_hi, const int32_t* pairs, int32_t n_pairs,
                    int64_t n_episodes, uint64_t seed, const float* ext_logits, float* obs,
                    int8_t* action, float* reward, float* logits, int n_threads) {
    const int N = 2, in = 11, A = 5;
    int64_t per = n_envs / n_pairs;
    int64_t W = env_hi - env_lo;
    parallel_for(W * n_episodes, n_threads, [&](int64_t job) {
        int64_t ep = job / W, e = env_lo + job % W;
        int64_t row = e / per;
        SpeakerListener sl;
        uint64_t g = (uint64_t)ep * (uint64_t)n_envs + (uint64_t)e;
        sl_reset(sl, g, seed);
        for (int t = 0; t < T; ++t) {
            int act[2];
            for (int i = 0; i < N; ++i) {
                int64_t idx = ((ep * T + t) * W + (e - env_lo)) * N + i;
                float o[11], lg[8];
                sl_obs(sl, i, o);
                Mlp m{params[pairs[row * N + i]], in, h1, h2, A, bf16};
                mlp_logits(m, o, lg);
                uint8_t legal[8] = {1, 1, 1, 1, 1, 1, 1, 1};
                if (i == 0) legal[3] = legal[4] = 0;          // the speaker only speaks
                float u = uniform24(draw(g, (uint32_t)t, (uint32_t)i, seed).x[0]);
                act[i] = sample_masked(ext_logits ? ext_logits + idx * A : lg, legal, A, u);
                if (obs) std::memcpy(obs + idx * in, o, sizeof(float) * in);
                if (logits) std::memcpy(logits + idx * A, lg, sizeof(float) * A);
                if (action) action[idx] = (int8_t)act[i];
            }
            float r[2];
            sl_step(sl, act, r);
            if (reward)
                for (int i = 0; i < N; ++i) reward[((ep * T + t) * W + (e - env_lo)) * N + i] = r[i];
        }
    });
}

// ---- Simple push and simple tag ----
// state: px,py,vx,vy of the agents, then lx,ly of the landmarks / obstacles
// (push [4*2 + 2] = 10 floats, tag [4*4 + 2*2] = 20 floats).
static void sc_load(const float* state, int N, int L, Spread& s) {
    s.N = N; s.L = L;
    for (int i = 0; i < N; ++i) {
        s.px[i] = state[4 * i]; s.py[i] = state[4 * i + 1];
        s.vx[i] = state[4 * i + 2]; s.vy[i] = state[4 * i + 3];
    }
    for (int l = 0; l < L; ++l) { s.lx[l] = state[4 * N + 2 * l]; s.ly[l] = state[4 * N + 2 * l + 1]; }
}
static void sc_store(const Spread& s, float* state) {
    for (int i = 0; i < s.N; ++i) {
        state[4 * i] = s.px[i]; state[4 * i + 1] = s.py[i];
        state[4 * i + 2] = s.vx[i]; state[4 * i + 3] = s.vy[i];
    }
    for (int l = 0; l < s.L; ++l) { state[4 * s.N + 2 * l] = s.lx[l]; state[4 * s.N + 2 * l + 1] = s.ly[l]; }
}

void orc_push_reset(uint64_t g, uint64_t seed, float* state) {
    Push a;
    push_reset(a, g, seed);
    sc_store(a.s, state);
}
void orc_push_step(float* state, const int32_t* action, float* reward) {
    Push a;
    sc_load(state, 2, 1, a.s);
    push_step(a, action, reward);
    sc_store(a.s, state);
}
void orc_push_obs(const float* state, float* obs /*[2][8]*/) {
    Push a;
    sc_load(state, 2, 1, a.s);
    for (int i = 0; i < 2; ++i) push_obs(a, i, obs + i * 8);
}
void orc_push_rollout(const float* const* params, int h1, int h2, int bf16, int T, int64_t n_envs,
                      int64_t env_lo, int64_t env_hi, const int32_t* pairs, int32_t n_pairs,
                      int64_t n_episodes, uint64_t seed, const float* ext_logits, float* obs,
                      int8_t* action, float* reward, float* logits, int n_threads) {
    scenario_rollout<PushEnvDef>(params, h1, h2, bf16, T, n_envs, env_lo, env_hi, pairs, n_pairs,
                                 n_episodes, seed, ext_logits, obs, action, reward, logits, n_threads);
}

void orc_tag_reset(uint64_t g, uint64_t seed, float* state) {
    Tag a;
    tag_reset(a, g, seed);
    sc_store(a.s, state);
}
void orc_tag_step(float* state, const int32_t* action, float* reward) {
    Tag a;
    sc_load(state, 4, 2, a.s);
    tag_step(a, action, reward);
    sc_store(a.s, state);
}
void orc_tag_obs(const float* state, float* obs /*[4][16]*/) {
    Tag a;
    sc_load(state, 4, 2, a.s);
    for (int i = 0; i < 4; ++i) tag_obs(a, i, obs + i * 16);
}
void orc_tag_rollout(const float* const* params, int h1, int h2, int bf16, int T, int64_t n_envs,
                     int64_t env_lo, int64_t env_hi, const int32_t* pairs, int32_t n_pairs,
                     int64_t n_episodes, uint64_t seed, const float* ext_logits, float* obs,
                     int8_t* action, float* reward, float* logits, int n_threads) {
    scenario_rollout<TagEnvDef>(params, h1, h2, bf16, T, n_envs, env_lo, env_hi, pairs, n_pairs,
                                n_episodes, seed, ext_logits, obs, action, reward, logits, n_threads);
}

// ---- Simple reference ----
// state: px,py,vx,vy of the 2 agents, lx,ly of the 3 landmarks, the two goals
// and the two last messages (-1: none) as floats ([4*2 + 2*3 + 4] = 18).
static void ref_load(const float* st, Reference& a, float rho) {
    sc_load(st, 2, 3, a.s);
    a.goal[0] = (int)st[14]; a.goal[1] = (int)st[15];
    a.msg[0] = (int)st[16]; a.msg[1] = (int)st[17];
    a.rho = rho;
}
static void ref_store(const Reference& a, float* st) {
    sc_store(a.s, st);
    st[14] = (float)a.goal[0]; st[15] = (float)a.goal[1];
    st[16] = (float)a.msg[0]; st[17] = (float)a.msg[1];
}
void orc_ref_reset(uint64_t g, uint64_t seed, float* state) {
    Reference a;
    ref_reset(a, g, seed);
    ref_store(a, state);
}
void orc_ref_step(float* state, const int32_t* action, float* reward, float rho) {
    Reference a;
    ref_load(state, a, rho);
    ref_step(a, action, reward);
    ref_store(a, state);
}
void orc_ref_obs(const float* state, float* obs /*[2][14]*/) {
    Reference a;
    ref_load(state, a, 0.5f);
    for (int i = 0; i < 2; ++i) ref_obs(a, i, obs + i * 14);
}
void orc_ref_rollout(const float* const* params, int h1, int h2, int bf16, int T, int64_t n_envs,
                     int64_t env_lo, int64_t env_hi, const int32_t* pairs, int32_t n_pairs,
                     int64_t n_episodes, uint64_t seed, const float* ext_logits, float* obs,
                     int8_t* action, float* reward, float* logits, int n_threads, float rho) {
    RefEnvDef::rho = rho;
    scenario_rollout<RefEnvDef>(params, h1, h2, bf16, T, n_envs, env_lo, env_hi, pairs, n_pairs,
                                n_episodes, seed, ext_logits, obs, action, reward, logits, n_threads);
}

}  // extern "C"
