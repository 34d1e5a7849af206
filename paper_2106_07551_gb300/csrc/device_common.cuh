// Device-side building blocks shared by the rollout and evaluation kernels:
// counter-based sampling, the deterministic exp used by the masked softmax,
// bulk-copy (TMA, non-tensor) staging with bounded mbarrier waits, and
// error flags. Written for sm_103a.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "internal.h"

namespace malib {

// ----------------------------------------------------------------------------
// Philox4x32-10 (Salmon et al., SC'11). Key = (seed lo32, seed hi32); counter
// layout used throughout: (episode id lo32, episode id hi32, step, agent), chance
// draws with agent = 0xFFFFFFFF (spread resets: step = entity index, landmarks
// offset by 0x80000000).
// ----------------------------------------------------------------------------
struct U4 { uint32_t x, y, z, w; };

__device__ __forceinline__ U4 philox10(uint32_t c0, uint32_t c1, uint32_t c2, uint32_t c3,
                                       uint32_t k0, uint32_t k1) {
#pragma unroll
    for (int r = 0; r < 10; ++r) {
        const uint32_t hi0 = __umulhi(0xD2511F53u, c0), lo0 = 0xD2511F53u * c0;
        const uint32_t hi1 = __umulhi(0xCD9E8D57u, c2), lo1 = 0xCD9E8D57u * c2;
        const uint32_t n0 = hi1 ^ c1 ^ k0;
        const uint32_t n2 = hi0 ^ c3 ^ k1;
        c0 = n0; c1 = lo1; c2 = n2; c3 = lo0;
        k0 += 0x9E3779B9u;
        k1 += 0xBB67AE85u;
    }
    return U4{c0, c1, c2, c3};
}

__device__ __forceinline__ U4 draw(uint64_t g, uint32_t step, uint32_t agent, uint64_t seed) {
    return philox10((uint32_t)g, (uint32_t)(g >> 32), step, agent, (uint32_t)seed,
                    (uint32_t)(seed >> 32));
}

constexpr uint32_t kChance = 0xFFFFFFFFu;

// [0,1) from the top 24 bits of a word (exact in fp32).
__device__ __forceinline__ float u24(uint32_t x) {
    return __uint2float_rn(x >> 8) * 5.9604644775390625e-08f;
}

// Index in [0, n) by multiply-shift.
__device__ __forceinline__ uint32_t pick(uint32_t x, uint32_t n) {
    return __umulhi(x, n);
}

// ----------------------------------------------------------------------------
// Deterministic exp: every step is one correctly-rounded IEEE operation (no
// contraction: explicit _rn intrinsics and fmaf), so that any implementation of
// the same steps gives the same bits. Cody-Waite reduction with ln2 split in a
// short head and a tail, Taylor polynomial of degree 7 (Horner, fused), 2^k
// from the exponent field. x <= -87 gives 0; x is clamped at 88.
// ----------------------------------------------------------------------------
__device__ __forceinline__ float det_expf(float x) {
    if (!(x > -87.0f)) return 0.0f;
    x = fminf(x, 88.0f);
    const float kf = rintf(__fmul_rn(x, 0x1.715476p+0f));
    float r = fmaf(-kf, 0x1.62e4p-1f, x);
    r = fmaf(-kf, 0x1.7f7d1cp-20f, r);
    float p = 0x1.a01a02p-13f;
    p = fmaf(p, r, 0x1.6c16c2p-10f);
    p = fmaf(p, r, 0x1.111112p-7f);
    p = fmaf(p, r, 0x1.555556p-5f);
    p = fmaf(p, r, 0x1.555556p-3f);
    p = fmaf(p, r, 0.5f);
    p = fmaf(p, r, 1.0f);
    p = fmaf(p, r, 1.0f);
    const int k = __float2int_rn(kf);
    return __fmul_rn(p, __int_as_float((k + 127) << 23));
}

// Masked softmax + inverse-CDF draw without division: m = max legal logit,
// e_a = det_expf(l_a - m) (0 if illegal), S = sum in ascending a, pick the first
// legal a with u*S < running sum; if rounding leaves none, the last legal a.
template <int A>
__device__ __forceinline__ int sample_masked(const float (&lg)[A], unsigned legal_bits, float u) {
    int first = -1;
#pragma unroll
    for (int a = A - 1; a >= 0; --a)
        if (legal_bits & (1u << a)) first = a;
    if (first < 0) return -1;
    float m = lg[first];
#pragma unroll
    for (int a = 0; a < A; ++a)
        if ((legal_bits & (1u << a)) && a > first && lg[a] > m) m = lg[a];
    float e[A];
    float S = 0.0f;
#pragma unroll
    for (int a = 0; a < A; ++a) {
        e[a] = (legal_bits & (1u << a)) ? det_expf(__fsub_rn(lg[a], m)) : 0.0f;
        S = __fadd_rn(S, e[a]);
    }
    const float thr = __fmul_rn(u, S);
    float C = 0.0f;
    int last = first, pickd = -1;
#pragma unroll
    for (int a = 0; a < A; ++a) {
        if (!(legal_bits & (1u << a))) continue;
        C = __fadd_rn(C, e[a]);
        last = a;
        if (pickd < 0 && thr < C) pickd = a;
    }
    return pickd >= 0 ? pickd : last;
}

// ----------------------------------------------------------------------------
// Bulk async copy global -> shared (the non-tensor TMA path) completing on an
// mbarrier, and bounded waits. Sizes and addresses must be 16-byte multiples.
// ----------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count)
                 : "memory");
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
                 "r"(bytes)
                 : "memory");
}

// Plain arrival (release at CTA scope) on a local mbarrier.
__device__ __forceinline__ void mbar_arrive_release(uint64_t* bar) {
    asm volatile("mbarrier.arrive.release.cta.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar))
                 : "memory");
}

// Shared -> global bulk copy (16-byte aligned addresses, size a multiple of
// 16), tracked by the issuing thread's bulk groups.
__device__ __forceinline__ void bulk_s2g(void* dst_gmem, const void* src_smem, uint32_t bytes) {
    asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(dst_gmem),
                 "r"(smem_u32(src_smem)), "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// The issuing thread's committed bulk copies have finished reading shared memory.
__device__ __forceinline__ void bulk_wait_read() {
    asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
}
// The issuing thread's committed bulk copies have completed.
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

__device__ __forceinline__ void bulk_g2s(void* dst_smem, const void* src_gmem, uint32_t bytes,
                                         uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::
            "r"(smem_u32(dst_smem)),
        "l"(src_gmem), "r"(bytes), "r"(smem_u32(bar))
        : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
        " selp.u32 %0, 1, 0, p;\n}" : "=r"(ok) : "r"(smem_u32(bar)), "r"(parity) : "memory");
    return ok != 0;
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
    return t;
}

// Waits for the barrier phase with the given parity for at most `limit_ns`.
// Returns false on expiry.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t* bar, uint32_t parity,
                                                  uint64_t limit_ns) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = globaltimer_ns();
    while (true) {
        if (mbar_try_wait(bar, parity)) return true;
        if (globaltimer_ns() - t0 > limit_ns) return false;
    }
}

constexpr uint64_t kWaitLimitNs = 1000000000ull;   // 1 s: far above any staging copy

// Stages `bytes` (16-byte multiple) from global to shared with one elected
// thread issuing bulk copies of at most 64 KB each; every thread then waits on
// the barrier phase `parity` (bounded). On expiry raises ERRBIT_TIMEOUT,
// waits once more (bounded) for the copies in flight, and returns false.
__device__ __forceinline__ bool stage_to_smem(void* dst, const void* src, uint32_t bytes,
                                              uint64_t* bar, uint32_t parity, int* err) {
    if (threadIdx.x == 0) {
        fence_proxy_async_smem();
        mbar_arrive_expect_tx(bar, bytes);
        uint32_t off = 0;
        while (off < bytes) {
            const uint32_t n = (bytes - off) < 65536u ? (bytes - off) : 65536u;
            bulk_g2s((char*)dst + off, (const char*)src + off, n, bar);
            off += n;
        }
    }
    if (!mbar_wait_bounded(bar, parity, kWaitLimitNs)) {
        atomicOr(err, ERRBIT_TIMEOUT);
        mbar_wait_bounded(bar, parity, kWaitLimitNs);
        return false;
    }
    return true;
}

// Warp-level inclusive sum helpers.
__device__ __forceinline__ long long warp_sum_ll(long long v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// One payoff-table row from a pair's integer sums over n hands (Sec. 3.2, the
// Monte-Carlo mean per combination): mean, standard error of the mean (sample
// variance with n - 1, clamped at 0), and the two sums as doubles. Correctly
// rounded double operations, so every caller writes the same bits.
__device__ __forceinline__ void finalize_pair(long long s1, long long s2, int64_t n, double* row) {
    const double dn = (double)n, d1 = (double)s1, d2 = (double)s2;
    const double mean = __ddiv_rn(d1, dn);
    double se = 0.0;
    if (n >= 2) {
        const double q = __ddiv_rn(__dmul_rn(d1, d1), dn);
        double var = __ddiv_rn(__dsub_rn(d2, q), (double)(n - 1));
        if (var < 0.0) var = 0.0;
        se = __dsqrt_rn(__ddiv_rn(var, dn));
    }
    row[0] = mean;
    row[1] = se;
    row[2] = d1;
    row[3] = d2;
}

}  // namespace malib
