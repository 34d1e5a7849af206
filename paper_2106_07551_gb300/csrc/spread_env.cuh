// Cooperative particle spread (App. B.1) on the device, one environment per
// thread with its state in registers; shared by the fp32 and tensor-core
// rollout kernels. Every arithmetic step is an explicit correctly-rounded fp32
// operation so that any two implementations of these steps agree bit for bit.
#pragma once

#include "contact.cuh"
#include "device_common.cuh"

namespace malib {

template <int N>
struct SpreadEnv {
    float px[N], py[N], vx[N], vy[N], lx[N], ly[N];
};

template <int N>
__device__ __forceinline__ void spread_reset(SpreadEnv<N>& s, uint64_t g, uint64_t seed) {
#pragma unroll
    for (int i = 0; i < N; ++i) {
        const U4 d = draw(g, (uint32_t)i, kChance, seed);
        s.px[i] = __fsub_rn(__fmul_rn(u24(d.x), 2.0f), 1.0f);
        s.py[i] = __fsub_rn(__fmul_rn(u24(d.y), 2.0f), 1.0f);
        s.vx[i] = 0.f;
        s.vy[i] = 0.f;
    }
#pragma unroll
    for (int l = 0; l < N; ++l) {
        const U4 d = draw(g, 0x80000000u + (uint32_t)l, kChance, seed);
        s.lx[l] = __fsub_rn(__fmul_rn(u24(d.x), 2.0f), 1.0f);
        s.ly[l] = __fsub_rn(__fmul_rn(u24(d.y), 2.0f), 1.0f);
    }
}

// Observation of agent i: velocity, position, landmarks relative to the agent,
// the other agents relative to it (ascending), zeros up to the row stride.
template <int N, int XS>
__device__ __forceinline__ void spread_obs(const SpreadEnv<N>& s, int i, float* o) {
    int k = 0;
    o[k++] = s.vx[i];
    o[k++] = s.vy[i];
    o[k++] = s.px[i];
    o[k++] = s.py[i];
#pragma unroll
    for (int l = 0; l < N; ++l) {
        o[k++] = __fsub_rn(s.lx[l], s.px[i]);
        o[k++] = __fsub_rn(s.ly[l], s.py[i]);
    }
#pragma unroll
    for (int j = 0; j < N; ++j) {
        if (j == i) continue;
        o[k++] = __fsub_rn(s.px[j], s.px[i]);
        o[k++] = __fsub_rn(s.py[j], s.py[i]);
    }
    for (; k < XS; ++k) o[k] = 0.f;
}

// spread_obs for a run-time agent index: the same values and operations, with
// every register array indexed at compile time (selects instead of indexing).
template <int N, int XS>
__device__ __forceinline__ void spread_obs_dyn(const SpreadEnv<N>& s, int i, float* o) {
    float px = 0.f, py = 0.f, vx = 0.f, vy = 0.f;
#pragma unroll
    for (int j = 0; j < N; ++j)
        if (j == i) { px = s.px[j]; py = s.py[j]; vx = s.vx[j]; vy = s.vy[j]; }
    int k = 0;
    o[k++] = vx;
    o[k++] = vy;
    o[k++] = px;
    o[k++] = py;
#pragma unroll
    for (int l = 0; l < N; ++l) {
        o[k++] = __fsub_rn(s.lx[l], px);
        o[k++] = __fsub_rn(s.ly[l], py);
    }
#pragma unroll
    for (int m = 0; m < N - 1; ++m) {
        const float qx = m < i ? s.px[m] : s.px[m + 1];
        const float qy = m < i ? s.py[m] : s.py[m + 1];
        o[k++] = __fsub_rn(qx, px);
        o[k++] = __fsub_rn(qy, py);
    }
#pragma unroll
    for (; k < XS; ++k) o[k] = 0.f;
}


__device__ __forceinline__ float sqdist(float ax, float ay, float bx, float by) {
    const float dx = __fsub_rn(ax, bx), dy = __fsub_rn(ay, by);
    return __fadd_rn(__fmul_rn(dx, dx), __fmul_rn(dy, dy));
}

// |p_i - p_j| < 0.3 (two radii of 0.15) with |.| the correctly rounded fp32
// square root of the squared distance holds exactly when the squared distance
// is below this threshold: the rounded square root is monotone, and the
// smallest fp32 value whose rounded root reaches 0.3f is fp32(0.3f * 0.3f).
constexpr float kCollideSq = 0x1.70a3d8p-4f;

// Mass 1, dt 0.1, damping 0.25, unit force along the chosen axis; reward after
// the move; collision when centres are closer than 2 x 0.15. local_ratio < 0:
// r_i = -(cover + coll_i); otherwise -((1 - local_ratio) cover + local_ratio
// coll_i), each operation rounded in the order written. The rounded
// square root is monotone, so the minimum over agents of the rounded distances
// to a landmark equals the rounded root of the minimum squared distance: one
// root per landmark gives the same bits as one per (landmark, agent).
// kContact: the agents (disks of radius 0.15) also push each other apart with
// the soft contact forces (contact.cuh), taken from the positions before the
// move and added to the action forces; landmarks do not collide.
template <int N, bool kContact = false>
__device__ __forceinline__ void spread_step(SpreadEnv<N>& s, const int (&act)[N], float (&r)[N],
                                            float local_ratio) {
    float Fx[N], Fy[N];
#pragma unroll
    for (int i = 0; i < N; ++i) unit_force(act[i], Fx[i], Fy[i]);
    if constexpr (kContact) {
        float rad[N];
#pragma unroll
        for (int i = 0; i < N; ++i) rad[i] = 0.15f;
        add_contacts<N, 0>(s.px, s.py, rad, nullptr, nullptr, nullptr, Fx, Fy);
    }
#pragma unroll
    for (int i = 0; i < N; ++i) {
        s.vx[i] = __fadd_rn(__fmul_rn(s.vx[i], 0.75f), __fmul_rn(Fx[i], 0.1f));
        s.vy[i] = __fadd_rn(__fmul_rn(s.vy[i], 0.75f), __fmul_rn(Fy[i], 0.1f));
        s.px[i] = __fadd_rn(s.px[i], __fmul_rn(s.vx[i], 0.1f));
        s.py[i] = __fadd_rn(s.py[i], __fmul_rn(s.vy[i], 0.1f));
    }
    float cover = 0.f;
#pragma unroll
    for (int l = 0; l < N; ++l) {
        float best = sqdist(s.px[0], s.py[0], s.lx[l], s.ly[l]);
#pragma unroll
        for (int j = 1; j < N; ++j) {
            const float d = sqdist(s.px[j], s.py[j], s.lx[l], s.ly[l]);
            best = d < best ? d : best;
        }
        cover = __fadd_rn(cover, __fsqrt_rn(best));
    }
    int coll[N];
#pragma unroll
    for (int i = 0; i < N; ++i) coll[i] = 0;
#pragma unroll
    for (int i = 0; i < N; ++i)
#pragma unroll
        for (int j = i + 1; j < N; ++j)
            if (sqdist(s.px[i], s.py[i], s.px[j], s.py[j]) < kCollideSq) { ++coll[i]; ++coll[j]; }
#pragma unroll
    for (int i = 0; i < N; ++i)
        r[i] = local_ratio < 0.f
                   ? -__fadd_rn(cover, (float)coll[i])
                   : -__fadd_rn(__fmul_rn(__fsub_rn(1.f, local_ratio), cover),
                                __fmul_rn(local_ratio, (float)coll[i]));
}

}  // namespace malib
