// Simple speaker listener (App. B.1) on the device, one environment per thread
// with its state in registers: agent 0 is the speaker, which does not move and
// whose action 0..2 is the message it sends (its actions 3 and 4 are not
// legal); agent 1 the listener, which moves with the spread dynamics and cannot
// speak; three landmarks, one of them the target. The listener sees the
// message sent at the previous step; both agents are rewarded by the
// listener's distance to the target. Every arithmetic step is an explicit
// correctly-rounded fp32 operation.
#pragma once

#include "device_common.cuh"
#include "spread_env.cuh"

namespace malib {

struct SlEnv {
    float px[2], py[2], vx[2], vy[2], lx[3], ly[3];
    int target;
    int msg;            // -1: none yet
};

constexpr int kSlObs = 11;
constexpr unsigned kSlSpeakerLegal = 0x7u;   // messages 0..2

// Agents and landmarks as in the spread reset (same chance counters); the
// target is pick(x, 3) of the chance draw with step field 0xC0000000.
__device__ __forceinline__ void sl_reset(SlEnv& s, uint64_t g, uint64_t seed) {
#pragma unroll
    for (int i = 0; i < 2; ++i) {
        const U4 d = draw(g, (uint32_t)i, kChance, seed);
        s.px[i] = __fsub_rn(__fmul_rn(u24(d.x), 2.0f), 1.0f);
        s.py[i] = __fsub_rn(__fmul_rn(u24(d.y), 2.0f), 1.0f);
        s.vx[i] = 0.f;
        s.vy[i] = 0.f;
    }
#pragma unroll
    for (int l = 0; l < 3; ++l) {
        const U4 d = draw(g, 0x80000000u + (uint32_t)l, kChance, seed);
        s.lx[l] = __fsub_rn(__fmul_rn(u24(d.x), 2.0f), 1.0f);
        s.ly[l] = __fsub_rn(__fmul_rn(u24(d.y), 2.0f), 1.0f);
    }
    s.target = (int)pick(draw(g, 0xC0000000u, kChance, seed).x, 3);
    s.msg = -1;
}

// Observation of agent i (compile-time), zeros up to the row stride XS:
// speaker - one-hot of the target; listener - velocity, landmarks - p_1
// (ascending), one-hot of the last message.
template <int XS>
__device__ __forceinline__ void sl_obs(const SlEnv& s, int i, float* o) {
#pragma unroll
    for (int k = 0; k < XS; ++k) o[k] = 0.f;
    if (i == 0) {
#pragma unroll
        for (int l = 0; l < 3; ++l) o[l] = s.target == l ? 1.f : 0.f;
        return;
    }
    o[0] = s.vx[1];
    o[1] = s.vy[1];
#pragma unroll
    for (int l = 0; l < 3; ++l) {
        o[2 + 2 * l] = __fsub_rn(s.lx[l], s.px[1]);
        o[3 + 2 * l] = __fsub_rn(s.ly[l], s.py[1]);
    }
#pragma unroll
    for (int m = 0; m < 3; ++m) o[8 + m] = s.msg == m ? 1.f : 0.f;
}

// The speaker's message, the listener's move (mass 1, dt 0.1, damping 0.25,
// unit force), then r_0 = r_1 = -d(p_1, target).
__device__ __forceinline__ void sl_step(SlEnv& s, const int (&act)[2], float (&r)[2]) {
    s.msg = act[0];
    const float fx = act[1] == 1 ? 1.f : (act[1] == 2 ? -1.f : 0.f);
    const float fy = act[1] == 3 ? 1.f : (act[1] == 4 ? -1.f : 0.f);
    s.vx[1] = __fadd_rn(__fmul_rn(s.vx[1], 0.75f), __fmul_rn(fx, 0.1f));
    s.vy[1] = __fadd_rn(__fmul_rn(s.vy[1], 0.75f), __fmul_rn(fy, 0.1f));
    s.px[1] = __fadd_rn(s.px[1], __fmul_rn(s.vx[1], 0.1f));
    s.py[1] = __fadd_rn(s.py[1], __fmul_rn(s.vy[1], 0.1f));
    const float tx = s.target == 0 ? s.lx[0] : (s.target == 1 ? s.lx[1] : s.lx[2]);
    const float ty = s.target == 0 ? s.ly[0] : (s.target == 1 ? s.ly[1] : s.ly[2]);
    const float d = __fsqrt_rn(sqdist(s.px[1], s.py[1], tx, ty));
    r[0] = -d;
    r[1] = -d;
}

}  // namespace malib
