// Simple push (App. B.1) on the device, one environment per thread with its
// state in registers: agent 0 is the adversary, agent 1 the good agent, one
// landmark. The two agents are disks of radius 0.15 that push each other with
// the soft contact forces (contact.cuh; the landmark does not collide). The
// good agent is rewarded for being close to the landmark, the adversary for
// being close to it while the good agent is far (the difference of the two
// distances). Every arithmetic step is an explicit correctly-rounded fp32
// operation.
#pragma once

#include "contact.cuh"
#include "device_common.cuh"
#include "spread_env.cuh"

namespace malib {

struct PushEnv {
    float px[2], py[2], vx[2], vy[2], lx, ly;
};

constexpr int kPushObs = 8;

// Agents and the landmark as in the spread reset (same chance counters).
__device__ __forceinline__ void push_reset(PushEnv& s, uint64_t g, uint64_t seed) {
#pragma unroll
    for (int i = 0; i < 2; ++i) {
        const U4 d = draw(g, (uint32_t)i, kChance, seed);
        s.px[i] = __fsub_rn(__fmul_rn(u24(d.x), 2.0f), 1.0f);
        s.py[i] = __fsub_rn(__fmul_rn(u24(d.y), 2.0f), 1.0f);
        s.vx[i] = 0.f;
        s.vy[i] = 0.f;
    }
    const U4 d = draw(g, 0x80000000u, kChance, seed);
    s.lx = __fsub_rn(__fmul_rn(u24(d.x), 2.0f), 1.0f);
    s.ly = __fsub_rn(__fmul_rn(u24(d.y), 2.0f), 1.0f);
}

// Observation of agent i (compile-time): velocity, position, landmark - p_i,
// the other agent - p_i, zeros up to the row stride XS.
template <int XS>
__device__ __forceinline__ void push_obs(const PushEnv& s, int i, float* o) {
    const int j = 1 - i;
    o[0] = s.vx[i];
    o[1] = s.vy[i];
    o[2] = s.px[i];
    o[3] = s.py[i];
    o[4] = __fsub_rn(s.lx, s.px[i]);
    o[5] = __fsub_rn(s.ly, s.py[i]);
    o[6] = __fsub_rn(s.px[j], s.px[i]);
    o[7] = __fsub_rn(s.py[j], s.py[i]);
#pragma unroll
    for (int k = kPushObs; k < XS; ++k) o[k] = 0.f;
}

// Unit action forces plus the pair's contact force (from the positions before
// the move); mass 1, dt 0.1, damping 0.25. Then, with d_i = |p_i - landmark|:
// r_0 = d_1 - d_0 (adversary), r_1 = -d_1 (good agent).
__device__ __forceinline__ void push_step(PushEnv& s, const int (&act)[2], float (&r)[2]) {
    float Fx[2], Fy[2];
    unit_force(act[0], Fx[0], Fy[0]);
    unit_force(act[1], Fx[1], Fy[1]);
    const float rad[2] = {0.15f, 0.15f};
    add_contacts<2, 0>(s.px, s.py, rad, nullptr, nullptr, nullptr, Fx, Fy);
#pragma unroll
    for (int i = 0; i < 2; ++i) {
        s.vx[i] = __fadd_rn(__fmul_rn(s.vx[i], 0.75f), __fmul_rn(Fx[i], 0.1f));
        s.vy[i] = __fadd_rn(__fmul_rn(s.vy[i], 0.75f), __fmul_rn(Fy[i], 0.1f));
        s.px[i] = __fadd_rn(s.px[i], __fmul_rn(s.vx[i], 0.1f));
        s.py[i] = __fadd_rn(s.py[i], __fmul_rn(s.vy[i], 0.1f));
    }
    const float d0 = __fsqrt_rn(sqdist(s.px[0], s.py[0], s.lx, s.ly));
    const float d1 = __fsqrt_rn(sqdist(s.px[1], s.py[1], s.lx, s.ly));
    r[0] = __fsub_rn(d1, d0);
    r[1] = -d1;
}

}  // namespace malib
