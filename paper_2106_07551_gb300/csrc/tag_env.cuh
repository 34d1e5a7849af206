// Simple tag (App. B.1) on the device, one environment per thread with its
// state in registers: agents 0..2 are the adversaries (radius 0.075, action
// force 3, speed limit 1.0), agent 3 the faster good agent (radius 0.05, action
// force 4, speed limit 1.3), two immovable obstacles (radius 0.2). All agents
// and obstacles collide with the soft contact forces (contact.cuh). An
// adversary hits the good agent when their centres are closer than 0.075 +
// 0.05; each hit costs the good agent 10 and pays every adversary 10. Every
// arithmetic step is an explicit correctly-rounded fp32 operation.
#pragma once

#include "contact.cuh"
#include "device_common.cuh"
#include "spread_env.cuh"

namespace malib {

struct TagEnv {
    float px[4], py[4], vx[4], vy[4], ox[2], oy[2];
};

constexpr int kTagObs = 16;

__device__ __forceinline__ float tag_radius(int i) { return i < 3 ? 0.075f : 0.05f; }
__device__ __forceinline__ float tag_accel(int i) { return i < 3 ? 3.0f : 4.0f; }
__device__ __forceinline__ float tag_vmax(int i) { return i < 3 ? 1.0f : 1.3f; }

// Agents and obstacles as in the spread reset (same chance counters; the
// obstacles take the landmark slots).
__device__ __forceinline__ void tag_reset(TagEnv& s, uint64_t g, uint64_t seed) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const U4 d = draw(g, (uint32_t)i, kChance, seed);
        s.px[i] = __fsub_rn(__fmul_rn(u24(d.x), 2.0f), 1.0f);
        s.py[i] = __fsub_rn(__fmul_rn(u24(d.y), 2.0f), 1.0f);
        s.vx[i] = 0.f;
        s.vy[i] = 0.f;
    }
#pragma unroll
    for (int l = 0; l < 2; ++l) {
        const U4 d = draw(g, 0x80000000u + (uint32_t)l, kChance, seed);
        s.ox[l] = __fsub_rn(__fmul_rn(u24(d.x), 2.0f), 1.0f);
        s.oy[l] = __fsub_rn(__fmul_rn(u24(d.y), 2.0f), 1.0f);
    }
}

// Observation of agent i (compile-time): velocity, position, obstacles - p_i,
// the other agents - p_i (ascending), then the good agent's velocity for an
// adversary (zeros for the good agent), zeros up to the row stride XS.
template <int XS>
__device__ __forceinline__ void tag_obs(const TagEnv& s, int i, float* o) {
    const float px = s.px[i], py = s.py[i];
    int k = 0;
    o[k++] = s.vx[i];
    o[k++] = s.vy[i];
    o[k++] = px;
    o[k++] = py;
#pragma unroll
    for (int l = 0; l < 2; ++l) {
        o[k++] = __fsub_rn(s.ox[l], px);
        o[k++] = __fsub_rn(s.oy[l], py);
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        if (j == i) continue;
        o[k++] = __fsub_rn(s.px[j], px);
        o[k++] = __fsub_rn(s.py[j], py);
    }
    o[k++] = i < 3 ? s.vx[3] : 0.f;
    o[k++] = i < 3 ? s.vy[3] : 0.f;
#pragma unroll
    for (; k < XS; ++k) o[k] = 0.f;
}

// Action forces (scaled by each agent's acceleration) plus the contact forces
// among the agents and from the obstacles, from the positions before the move;
// per agent v <- 0.75 v + 0.1 F, then v <- (v / |v|) vmax per component when
// |v| > vmax, then p <- p + 0.1 v. Rewards from the positions after the move.
__device__ __forceinline__ void tag_step(TagEnv& s, const int (&act)[4], float (&r)[4]) {
    float Fx[4], Fy[4], rad[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        float ux, uy;
        unit_force(act[i], ux, uy);
        Fx[i] = __fmul_rn(tag_accel(i), ux);
        Fy[i] = __fmul_rn(tag_accel(i), uy);
        rad[i] = tag_radius(i);
    }
    const float orad[2] = {0.2f, 0.2f};
    add_contacts<4, 2>(s.px, s.py, rad, s.ox, s.oy, orad, Fx, Fy);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        float vx = __fadd_rn(__fmul_rn(s.vx[i], 0.75f), __fmul_rn(Fx[i], 0.1f));
        float vy = __fadd_rn(__fmul_rn(s.vy[i], 0.75f), __fmul_rn(Fy[i], 0.1f));
        const float speed = __fsqrt_rn(__fadd_rn(__fmul_rn(vx, vx), __fmul_rn(vy, vy)));
        if (speed > tag_vmax(i)) {
            vx = __fmul_rn(__fdiv_rn(vx, speed), tag_vmax(i));
            vy = __fmul_rn(__fdiv_rn(vy, speed), tag_vmax(i));
        }
        s.vx[i] = vx;
        s.vy[i] = vy;
        s.px[i] = __fadd_rn(s.px[i], __fmul_rn(vx, 0.1f));
        s.py[i] = __fadd_rn(s.py[i], __fmul_rn(vy, 0.1f));
    }
    int hits = 0;
#pragma unroll
    for (int i = 0; i < 3; ++i)
        if (__fsqrt_rn(sqdist(s.px[i], s.py[i], s.px[3], s.py[3])) < __fadd_rn(tag_radius(i), tag_radius(3)))
            ++hits;
#pragma unroll
    for (int i = 0; i < 3; ++i) r[i] = __fmul_rn(10.0f, (float)hits);
    r[3] = __fmul_rn(-10.0f, (float)hits);
}

}  // namespace malib
