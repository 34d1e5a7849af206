// Simple adversary (App. B.1) on the device, one environment per thread with
// its state in registers: agent 0 is the adversary, agents 1 and 2 the good
// agents, two landmarks of which one is the target. The good agents are
// rewarded for being close to the target and for the adversary being far from
// it, the adversary (not told which landmark is the target) for being close to
// it. Every arithmetic step is an explicit correctly-rounded fp32 operation.
#pragma once

#include "device_common.cuh"
#include "spread_env.cuh"

namespace malib {

struct AdvEnv {
    float px[3], py[3], vx[3], vy[3], lx[2], ly[2];
    int target;
};

constexpr int kAdvObs = 14;

// Agents and landmarks as in the spread reset (same chance counters); the
// target is pick(x, 2) of the chance draw with step field 0xC0000000.
__device__ __forceinline__ void adv_reset(AdvEnv& s, uint64_t g, uint64_t seed) {
#pragma unroll
    for (int i = 0; i < 3; ++i) {
        const U4 d = draw(g, (uint32_t)i, kChance, seed);
        s.px[i] = __fsub_rn(__fmul_rn(u24(d.x), 2.0f), 1.0f);
        s.py[i] = __fsub_rn(__fmul_rn(u24(d.y), 2.0f), 1.0f);
        s.vx[i] = 0.f;
        s.vy[i] = 0.f;
    }
#pragma unroll
    for (int l = 0; l < 2; ++l) {
        const U4 d = draw(g, 0x80000000u + (uint32_t)l, kChance, seed);
        s.lx[l] = __fsub_rn(__fmul_rn(u24(d.x), 2.0f), 1.0f);
        s.ly[l] = __fsub_rn(__fmul_rn(u24(d.y), 2.0f), 1.0f);
    }
    s.target = (int)pick(draw(g, 0xC0000000u, kChance, seed).x, 2);
}

// Observation of agent i (compile-time): velocity, position, target - p_i
// (zeros for the adversary), landmarks - p_i, the other agents - p_i
// (ascending), zeros up to the row stride XS.
template <int XS>
__device__ __forceinline__ void adv_obs(const AdvEnv& s, int i, float* o) {
    const float px = s.px[i], py = s.py[i];
    const float tx = s.target ? s.lx[1] : s.lx[0], ty = s.target ? s.ly[1] : s.ly[0];
    int k = 0;
    o[k++] = s.vx[i];
    o[k++] = s.vy[i];
    o[k++] = px;
    o[k++] = py;
    o[k++] = i == 0 ? 0.f : __fsub_rn(tx, px);
    o[k++] = i == 0 ? 0.f : __fsub_rn(ty, py);
#pragma unroll
    for (int l = 0; l < 2; ++l) {
        o[k++] = __fsub_rn(s.lx[l], px);
        o[k++] = __fsub_rn(s.ly[l], py);
    }
#pragma unroll
    for (int j = 0; j < 3; ++j) {
        if (j == i) continue;
        o[k++] = __fsub_rn(s.px[j], px);
        o[k++] = __fsub_rn(s.py[j], py);
    }
#pragma unroll
    for (; k < XS; ++k) o[k] = 0.f;
}

// The spread dynamics (mass 1, dt 0.1, damping 0.25, unit force), then, with
// d(.) the distance to the target: r_0 = -d(p_0) and r_1 = r_2 =
// -min(d(p_1), d(p_2)) + d(p_0). The rounded square root is monotone, so the
// minimum of the rounded distances is the rounded root of the minimum square.
__device__ __forceinline__ void adv_step(AdvEnv& s, const int (&act)[3], float (&r)[3]) {
#pragma unroll
    for (int i = 0; i < 3; ++i) {
        const float fx = act[i] == 1 ? 1.f : (act[i] == 2 ? -1.f : 0.f);
        const float fy = act[i] == 3 ? 1.f : (act[i] == 4 ? -1.f : 0.f);
        s.vx[i] = __fadd_rn(__fmul_rn(s.vx[i], 0.75f), __fmul_rn(fx, 0.1f));
        s.vy[i] = __fadd_rn(__fmul_rn(s.vy[i], 0.75f), __fmul_rn(fy, 0.1f));
        s.px[i] = __fadd_rn(s.px[i], __fmul_rn(s.vx[i], 0.1f));
        s.py[i] = __fadd_rn(s.py[i], __fmul_rn(s.vy[i], 0.1f));
    }
    const float tx = s.target ? s.lx[1] : s.lx[0], ty = s.target ? s.ly[1] : s.ly[0];
    const float d_adv = __fsqrt_rn(sqdist(s.px[0], s.py[0], tx, ty));
    const float q1 = sqdist(s.px[1], s.py[1], tx, ty), q2 = sqdist(s.px[2], s.py[2], tx, ty);
    const float d_good = __fsqrt_rn(q1 < q2 ? q1 : q2);
    r[0] = -d_adv;
    r[1] = __fadd_rn(-d_good, d_adv);
    r[2] = r[1];
}

}  // namespace malib
