// Leduc hold'em rules on the device (registers only), shared by the fp32 and
// tensor-core evaluation kernels.
#pragma once

#include "device_common.cuh"

namespace malib {

// ---------------------------------------------------------------- Leduc
// Six cards (two each of J, Q, K; rank = card / 2), ante 1, two rounds with
// raise sizes 2 and 4, at most two raises a round, seat 0 first in both rounds,
// public card revealed in round 2. Actions: 0 fold, 1 call/check, 2 raise.
struct LeducHand {
    int c0, c1, pub;
    int round, con0, con1, raises, nact, actor, done, payoff;
    __device__ int con_of(int seat) const { return seat ? con1 : con0; }
    __device__ int card_of(int seat) const { return seat ? c1 : c0; }
};

__device__ __forceinline__ void leduc_deal(LeducHand& h, uint64_t g, uint64_t seed) {
    const U4 d = draw(g, 0, kChance, seed);
    const int c0 = (int)pick(d.x, 6);
    const int j = (int)pick(d.y, 5);
    const int c1 = j + (j >= c0 ? 1 : 0);
    const int lo = min(c0, c1), hi = max(c0, c1);
    int p = (int)pick(d.z, 4);
    if (p >= lo) ++p;
    if (p >= hi) ++p;
    h.c0 = c0; h.c1 = c1; h.pub = p;
    h.round = 0; h.con0 = 1; h.con1 = 1; h.raises = 0; h.nact = 0;
    h.actor = 0; h.done = 0; h.payoff = 0;
}

__device__ __forceinline__ unsigned leduc_legal(const LeducHand& h) {
    const int me = h.actor;
    return (h.con_of(1 - me) > h.con_of(me) ? 1u : 0u) | 2u | (h.raises < 2 ? 4u : 0u);
}

__device__ __forceinline__ void leduc_obs(const LeducHand& h, float (&o)[17]) {
    const int me = h.actor, op = 1 - me;
    const unsigned lg = leduc_legal(h);
    const int rank = h.card_of(me) >> 1;
    const int pubi = 3 + (h.round ? (h.pub >> 1) : 3);
#pragma unroll
    for (int i = 0; i < 3; ++i) o[i] = rank == i ? 1.f : 0.f;
#pragma unroll
    for (int i = 3; i < 7; ++i) o[i] = pubi == i ? 1.f : 0.f;
    o[7] = h.round == 0 ? 1.f : 0.f;
    o[8] = h.round == 1 ? 1.f : 0.f;
    o[9] = __fdiv_rn((float)h.con_of(me), 13.0f);
    o[10] = __fdiv_rn((float)h.con_of(op), 13.0f);
#pragma unroll
    for (int i = 0; i < 3; ++i) o[11 + i] = h.raises == i ? 1.f : 0.f;
    o[14] = (lg & 1u) ? 1.f : 0.f;
    o[15] = 1.f;
    o[16] = (lg & 4u) ? 1.f : 0.f;
}

__device__ __forceinline__ int leduc_showdown(const LeducHand& h) {
    const int r0 = h.c0 >> 1, r1 = h.c1 >> 1, rp = h.pub >> 1;
    int w;
    if (r0 == rp) w = 1;
    else if (r1 == rp) w = -1;
    else w = (r0 > r1) - (r0 < r1);
    return w > 0 ? h.con1 : (w < 0 ? -h.con0 : 0);
}

__device__ __forceinline__ void leduc_apply(LeducHand& h, int a) {
    const int me = h.actor, op = 1 - me;
    if (a == 0) {
        h.done = 1;
        h.payoff = me == 0 ? -h.con0 : h.con1;
        return;
    }
    ++h.nact;
    const int c_op = h.con_of(op);
    if (a == 2) {
        const int c = c_op + (h.round == 0 ? 2 : 4);
        if (me) h.con1 = c; else h.con0 = c;
        ++h.raises;
        h.actor = op;
        return;
    }
    if (me) h.con1 = c_op; else h.con0 = c_op;
    if (h.nact >= 2) {
        if (h.round == 0) {
            h.round = 1; h.raises = 0; h.nact = 0; h.actor = 0;
        } else {
            h.done = 1;
            h.payoff = leduc_showdown(h);
        }
    } else {
        h.actor = op;
    }
}

}  // namespace malib
