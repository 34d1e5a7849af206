// Collisions as forces between disks (App. B.1: agents that collide, obstacles
// that block the way), for the particle scenarios on the device. The paper
// gives no force law; the model is the soft contact of the particle
// environments it runs: for disks at a and b whose radii sum to dmin, with
// delta = a - b and d = |delta|, the overlap is smoothed by a softplus of
// margin k = 0.001,
//   pen = k log(1 + exp((dmin - d) / k)),
// and a feels F_c pen delta / d (F_c = 100), b its negative. Every step is one
// correctly rounded fp32 operation in a fixed order, so the forces are the same
// bits wherever these steps are evaluated.
#pragma once

#include "device_common.cuh"

namespace malib {

constexpr float kContactMargin = 0.001f;
constexpr float kContactForce = 100.0f;

// log(1 + y) for y in [0, 1]: 2 atanh(z) with z = y / (2 + y) <= 1/3, the odd
// series of atanh up to z^17 (the rest is below 2^-32 of the sum) in Horner
// form in z^2 with fused multiply-adds.
__device__ __forceinline__ float det_log1pf(float y) {
    if (!(y > 0.0f)) return 0.0f;
    const float z = __fdiv_rn(y, __fadd_rn(2.0f, y));
    const float w = __fmul_rn(z, z);
    float p = 0x1.e1e1e2p-5f;          // 1/17
    p = fmaf(p, w, 0x1.111112p-4f);    // 1/15
    p = fmaf(p, w, 0x1.3b13b2p-4f);    // 1/13
    p = fmaf(p, w, 0x1.745d18p-4f);    // 1/11
    p = fmaf(p, w, 0x1.c71c72p-4f);    // 1/9
    p = fmaf(p, w, 0x1.24924ap-3f);    // 1/7
    p = fmaf(p, w, 0x1.99999ap-3f);    // 1/5
    p = fmaf(p, w, 0x1.555556p-2f);    // 1/3
    p = fmaf(p, w, 1.0f);
    return __fmul_rn(__fmul_rn(2.0f, z), p);
}

// The force on disk a from disk b, in the order dx, dy, q = dx dx + dy dy,
// d = sqrt(q), x = (dmin - d) / k, softplus(x) = max(x, 0) + log1p(exp(-|x|)),
// pen = k softplus, c = (F_c pen) / d, (c dx, c dy). False (no force) when
// d = 0 or pen = 0 (the latter once d - dmin >= 87 k: det_expf gives 0).
__device__ __forceinline__ bool contact_force(float ax, float ay, float bx, float by, float dmin,
                                              float& fx, float& fy) {
    const float dx = __fsub_rn(ax, bx), dy = __fsub_rn(ay, by);
    const float d = __fsqrt_rn(__fadd_rn(__fmul_rn(dx, dx), __fmul_rn(dy, dy)));
    if (d == 0.0f) return false;
    const float x = __fdiv_rn(__fsub_rn(dmin, d), kContactMargin);
    const float sp = __fadd_rn(x > 0.0f ? x : 0.0f, det_log1pf(det_expf(-fabsf(x))));
    const float pen = __fmul_rn(kContactMargin, sp);
    if (pen == 0.0f) return false;
    const float c = __fdiv_rn(__fmul_rn(kContactForce, pen), d);
    fx = __fmul_rn(c, dx);
    fy = __fmul_rn(c, dy);
    return true;
}

// Adds to F the contact forces among N movable disks (pairs a < b ascending: a
// +f, b -f), then those of M immovable disks on each movable one (a ascending,
// then o ascending). A force is added only where one acts, so without contact
// F keeps its bits.
template <int N, int M>
__device__ __forceinline__ void add_contacts(const float (&px)[N], const float (&py)[N], const float (&rad)[N],
                                             const float* ox, const float* oy, const float* orad,
                                             float (&Fx)[N], float (&Fy)[N]) {
#pragma unroll
    for (int a = 0; a < N; ++a)
#pragma unroll
        for (int b = a + 1; b < N; ++b) {
            float fx, fy;
            if (contact_force(px[a], py[a], px[b], py[b], __fadd_rn(rad[a], rad[b]), fx, fy)) {
                Fx[a] = __fadd_rn(Fx[a], fx);
                Fy[a] = __fadd_rn(Fy[a], fy);
                Fx[b] = __fsub_rn(Fx[b], fx);
                Fy[b] = __fsub_rn(Fy[b], fy);
            }
        }
#pragma unroll
    for (int a = 0; a < N; ++a)
#pragma unroll
        for (int o = 0; o < M; ++o) {
            float fx, fy;
            if (contact_force(px[a], py[a], ox[o], oy[o], __fadd_rn(rad[a], orad[o]), fx, fy)) {
                Fx[a] = __fadd_rn(Fx[a], fx);
                Fy[a] = __fadd_rn(Fy[a], fy);
            }
        }
}

// Unit force of the five discrete actions (0 noop, 1 +x, 2 -x, 3 +y, 4 -y).
__device__ __forceinline__ void unit_force(int act, float& fx, float& fy) {
    fx = act == 1 ? 1.f : (act == 2 ? -1.f : 0.f);
    fy = act == 3 ? 1.f : (act == 4 ? -1.f : 0.f);
}

}  // namespace malib
