// Simple reference (App. B.1) on the device, one environment per thread with
// its state in registers: two agents, three landmarks; each agent's goal
// landmark is known only to the other agent, and both speak and move. An action
// is a move and a message at once, a = 5 * message + move (15 actions). The
// message an agent sends at step t reaches the other agent's observation at
// step t + 1. Rewards weight each agent's own distance to its goal against the
// average of both (local_ratio). Every arithmetic step is an explicit
// correctly-rounded fp32 operation.
#pragma once

#include "contact.cuh"
#include "device_common.cuh"
#include "spread_env.cuh"

namespace malib {

struct RefEnv {
    float px[2], py[2], vx[2], vy[2], lx[3], ly[3];
    int goal[2];
    int msg[2];           // -1: none yet
};

constexpr int kRefObs = 14, kRefActions = 15;

// Agents and landmarks as in the spread reset (same chance counters); agent
// i's goal is pick(x, 3) of the chance draw with step field 0xC0000000 + i.
__device__ __forceinline__ void ref_reset(RefEnv& s, uint64_t g, uint64_t seed) {
#pragma unroll
    for (int i = 0; i < 2; ++i) {
        const U4 d = draw(g, (uint32_t)i, kChance, seed);
        s.px[i] = __fsub_rn(__fmul_rn(u24(d.x), 2.0f), 1.0f);
        s.py[i] = __fsub_rn(__fmul_rn(u24(d.y), 2.0f), 1.0f);
        s.vx[i] = 0.f;
        s.vy[i] = 0.f;
        s.goal[i] = (int)pick(draw(g, 0xC0000000u + (uint32_t)i, kChance, seed).x, 3);
        s.msg[i] = -1;
    }
#pragma unroll
    for (int l = 0; l < 3; ++l) {
        const U4 d = draw(g, 0x80000000u + (uint32_t)l, kChance, seed);
        s.lx[l] = __fsub_rn(__fmul_rn(u24(d.x), 2.0f), 1.0f);
        s.ly[l] = __fsub_rn(__fmul_rn(u24(d.y), 2.0f), 1.0f);
    }
}

// Observation of agent i (compile-time): velocity, landmarks - p_i, the other
// agent's goal as a one-hot, the other agent's last message as a one-hot
// (zeros before the first), zeros up to the row stride XS.
template <int XS>
__device__ __forceinline__ void ref_obs(const RefEnv& s, int i, float* o) {
    const int j = 1 - i;
    o[0] = s.vx[i];
    o[1] = s.vy[i];
#pragma unroll
    for (int l = 0; l < 3; ++l) {
        o[2 + 2 * l] = __fsub_rn(s.lx[l], s.px[i]);
        o[3 + 2 * l] = __fsub_rn(s.ly[l], s.py[i]);
    }
#pragma unroll
    for (int q = 0; q < 3; ++q) {
        o[8 + q] = s.goal[j] == q ? 1.f : 0.f;
        o[11 + q] = s.msg[j] == q ? 1.f : 0.f;
    }
#pragma unroll
    for (int k = kRefObs; k < XS; ++k) o[k] = 0.f;
}

// The spread dynamics for both agents' moves, the messages stored, then with
// d_i = |p_i - goal_i| and rho the local ratio:
// r_i = -((1 - rho) ((d_0 + d_1) 0.5) + rho d_i).
__device__ __forceinline__ void ref_step(RefEnv& s, const int (&act)[2], float (&r)[2], float rho) {
#pragma unroll
    for (int i = 0; i < 2; ++i) {
        float fx, fy;
        unit_force(act[i] % 5, fx, fy);
        s.vx[i] = __fadd_rn(__fmul_rn(s.vx[i], 0.75f), __fmul_rn(fx, 0.1f));
        s.vy[i] = __fadd_rn(__fmul_rn(s.vy[i], 0.75f), __fmul_rn(fy, 0.1f));
        s.px[i] = __fadd_rn(s.px[i], __fmul_rn(s.vx[i], 0.1f));
        s.py[i] = __fadd_rn(s.py[i], __fmul_rn(s.vy[i], 0.1f));
        s.msg[i] = act[i] / 5;
    }
    float d[2];
#pragma unroll
    for (int i = 0; i < 2; ++i) {
        float gx = s.lx[0], gy = s.ly[0];
#pragma unroll
        for (int l = 1; l < 3; ++l)
            if (s.goal[i] == l) { gx = s.lx[l]; gy = s.ly[l]; }
        d[i] = __fsqrt_rn(sqdist(s.px[i], s.py[i], gx, gy));
    }
    const float mean = __fmul_rn(__fadd_rn(d[0], d[1]), 0.5f);
    const float shared = __fmul_rn(__fsub_rn(1.0f, rho), mean);
#pragma unroll
    for (int i = 0; i < 2; ++i) r[i] = -__fadd_rn(shared, __fmul_rn(rho, d[i]));
}

}  // namespace malib
