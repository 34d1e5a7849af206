// Pipelined bf16 policy forward on the 5th-generation tensor cores: a stream of
// 128-row observation tiles through one resident policy
//   logits = W3 relu(W2 relu(W1 x + b1) + b2) + b3
// (bf16 weights and layer inputs, fp32 accumulation), with two tiles in flight
// so that the tensor pipe runs one tile's MMAs while the epilogue warps convert
// the other tile's accumulator.
//
// Tensor memory (512 columns) is two slots; tile t uses slot t mod 2, columns
// H = [256 s, 256 s + 128) and ACC = [256 s + 128, 256 s + 256). Each tile runs
// three MMA groups (N = 128, M = 128 rows) in its slot, each followed by an
// epilogue:
//   G0  ACC = X W1[0:128]^T, H = X W1[128:256]^T (fp32)
//       ep: h1 = bf16(relu(. + b1)), packed two per 32-bit column (lower k in
//       the low half, row i in lane i) into H, each warp within the columns it
//       read: neurons 128 + 32B .. + 32 at H[32B, 32B + 16) and neurons 32B ..
//       + 32 at H[32B + 16, 32B + 32), B = 0..3
//   G1  ACC = h1 W2[0:128]^T       G2  ACC = h1 W2[128:256]^T
//       ep: h2 = bf16(relu(ACC + b2)) is read in the mma.sync fragment layout
//       (tcgen05.ld 16x256b) and layer 3 runs on it as warp-level MMAs
//       (m16n8k16, W3 as the B operand, actions padded to 8), accumulating each
//       warp's partial logits over its neurons in registers; after G2 the
//       partials of a row (one per warp of its lane quarter) go to shared
//       memory, where the consumer adds them and b3.
// Layer 3 is 0.4 % of the flops; as tcgen05 MMAs of N = 16 it cost as much
// tensor-pipe time as half of layer 2, so it runs on the warp-level path.
//
// Roles: each slot has its own epilogue team of TW warps (warps TW s .. TW s +
// TW - 1; in a team, warp w handles lane quarter w % 4 and, with TW = 8, half
// w / 4 of the columns), so the two slots' epilogues run concurrently; the
// first thread of warp 2 TW + s issues slot s's MMAs, each group as soon as it
// is ready. The kernel supplies the tiles (producers: X(t) into buffer
// t % kNX, then one arrival on x_full) and takes the results (consumers: after
// p_full of slot t % 2, partial logits [TW / 4][128][A] fp32, then one arrival
// on p_free). Each mbarrier is waited on in
// strict phase order, so parities are counted, never guessed; every wait is
// bounded (a timeout raises ERRBIT_TIMEOUT and marks the engine dead, after
// which no role waits again).
#pragma once

#include <cstdint>

#include "device_common.cuh"
#include "tc_common.cuh"

namespace malib {

__device__ __forceinline__ bool mbar_test_wait(uint64_t* bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n"
        " selp.u32 %0, 1, 0, p;\n}" : "=r"(ok) : "r"(smem_u32(bar)), "r"(parity) : "memory");
    return ok != 0;
}

// D (+)= A B, m16n8k16, bf16 inputs, fp32 accumulation (warp-level MMA).
__device__ __forceinline__ void mma_m16n8k16(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                             uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
        "{%8, %9}, {%0, %1, %2, %3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

template <int K1, int A, int NX = 3, int TW = 8>
struct Eng2 {
    static_assert(K1 % 16 == 0 && K1 <= 48 && A >= 1 && A <= 8, "shapes built");
    static_assert(TW == 4 || TW == 8, "epilogue team of 4 or 8 warps");
    // ---- the policy in shared memory: the leading part of its global image
    // (tc_image_bytes layout), staged once
    static constexpr uint32_t kW1 = 0;                          // bf16 [256][K1], core-matrix K-major
    static constexpr uint32_t kW2 = 256u * K1 * 2;              // bf16 [256][256]
    static constexpr uint32_t kW3 = kW2 + 256u * 256 * 2;       // bf16 [16][256]
    static constexpr uint32_t kB1 = kW3 + 16u * 256 * 2;        // fp32 b1 [256]
    static constexpr uint32_t kB2 = kB1 + 1024;                 // fp32 b2 [256]
    static constexpr uint32_t kB3 = kB2 + 1024;                 // fp32 b3 [16]
    static constexpr uint32_t kImage = kB3 + 64;                // bytes staged
    static constexpr uint32_t kXBytes = 128u * K1 * 2;          // one observation tile
    static constexpr int kTeamWarps = TW;                       // epilogue warps per slot
    static constexpr int kSplit = TW / 4;                       // column parts of a lane quarter
    static constexpr uint32_t kPBytes = kSplit * 128u * A * 4;  // one slot's partials [kSplit][128][A]
    static constexpr uint32_t kLboX = 16 * 128;                 // K-chunk stride, 128 rows
    static constexpr uint32_t kLboW = 32 * 128;                 // K-chunk stride, 256 rows
    static constexpr int kNX = NX;
    static constexpr uint32_t kTmemCols = 512;
    static constexpr int kEpiWarps = 2 * TW;                    // two teams
    static constexpr int kTeamThreads = 32 * TW;
    static constexpr int kIssuerWarp = kEpiWarps;               // this warp and the next
    static constexpr int kOps = 3;                              // MMA groups per tile

    // Shared-memory state of the engine (the kernel places one instance in
    // static shared memory and calls init() from one thread).
    struct Bars {
        uint64_t stage;               // policy staged (tx bytes)
        uint64_t acc_full[2];         // a slot's MMA group complete (tcgen05.commit)
        uint64_t ep_done[2];          // a slot's epilogue of that group complete (its team's threads)
        uint64_t x_full[NX];          // tile's observations written (1 arrival)
        uint64_t x_free[NX];          // tile's layer 1 complete (tcgen05.commit)
        uint64_t p_full[2];           // slot's partial logits written (one arrival per team warp)
        uint64_t p_free[2];           // slot's partials read by the consumers (1 arrival)
        uint64_t drained[2];          // every MMA a slot's thread issued complete (tcgen05.commit)
        uint32_t dead;                // a bounded wait expired: nobody waits any more
        __device__ void init() {
            mbar_init(&stage, 1);
            for (int s = 0; s < 2; ++s) {
                mbar_init(&acc_full[s], 1);
                mbar_init(&ep_done[s], kTeamThreads);
                mbar_init(&p_full[s], TW);
                mbar_init(&p_free[s], 1);
            }
            for (int b = 0; b < NX; ++b) {
                mbar_init(&x_full[b], 1);
                mbar_init(&x_free[b], 1);
            }
            mbar_init(&drained[0], 1);
            mbar_init(&drained[1], 1);
            dead = 0u;
        }
    };

    __device__ static bool is_dead(Bars& b) { return *(volatile uint32_t*)&b.dead != 0u; }
    __device__ static void mark_dead(Bars& b, int* err) {
        *(volatile uint32_t*)&b.dead = 1u;
        atomicOr(err, ERRBIT_TIMEOUT);
    }

    // Bounded wait that marks the engine dead on expiry (and skips once dead).
    __device__ static bool wait(Bars& b, uint64_t* bar, uint32_t parity, int* err) {
        if (is_dead(b)) return false;
        if (mbar_wait_bounded(bar, parity, kWaitLimitNs)) return true;
        mark_dead(b, err);
        return false;
    }
    // The same by polling, without suspending the thread (for the MMA thread,
    // which has nothing else to do and must react at once).
    __device__ static bool spin(Bars& b, uint64_t* bar, uint32_t parity, int* err) {
        if (mbar_test_wait(bar, parity)) return true;
        const uint64_t t0 = globaltimer_ns();
        while (!mbar_test_wait(bar, parity)) {
            if (is_dead(b)) return false;
            if (globaltimer_ns() - t0 > kWaitLimitNs) {
                mark_dead(b, err);
                return false;
            }
        }
        return true;
    }

    // Stages a policy image from global memory (one thread); completes on
    // b.stage, which the users wait on (phase parity = stagings so far & 1).
    __device__ static void stage(uint8_t* smem, const uint8_t* gimg, Bars& b) {
        fence_proxy_async_smem();
        mbar_arrive_expect_tx(&b.stage, kImage);
        for (uint32_t off = 0; off < kImage; off += 32768u)
            bulk_g2s(smem + off, gimg + off, min(32768u, kImage - off), &b.stage);
    }

    // Byte offset of the 8 bf16 inputs k..k+7 of a row in an observation tile.
    __device__ static uint32_t x_offset(int row, int k) { return tc::cm_offset(row, k, 128, 2); }

    // Column of H holding the packed h1 inputs 16 k .. 16 k + 15 of layer 2.
    __device__ static uint32_t h1_col(int k) {
        return k < 8 ? 32u * (uint32_t)(k >> 1) + 16u + 8u * (uint32_t)(k & 1)
                     : 32u * (uint32_t)((k - 8) >> 1) + 8u * (uint32_t)(k & 1);
    }

    __device__ static void mma_ts(uint32_t d, uint32_t a_tmem, uint64_t b, uint32_t idesc, bool acc) {
        asm volatile(
            "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
            " tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n}" ::"r"(d),
            "r"(a_tmem), "l"(b), "r"(idesc), "r"((uint32_t)acc)
            : "memory");
    }

    struct Slot {
        uint32_t total = 0;           // groups handled in this slot over all runs
    };

    // ------------------------------------------------------------------ issuer
    // The MMA-issuing thread of slot S (the first thread of warp 16 + S). A
    // thread that issues tcgen05.mma is held until its MMAs have nearly
    // completed, so each slot has its own: while one is held by its group, the
    // other's next group is already queued on the tensor pipe, and each
    // thread's commits track only its own MMAs. Tiles are numbered t = 0, 1,
    // ... over the whole kernel; run(n) issues the slot's groups of tiles
    // t .. t + n - 1 (those of its parity).
    template <int S>
    struct Issuer {
        uint32_t t = 0;               // first tile of the next run
        Slot sl;

        // Group `op` of tile tt once the slot's previous group has been
        // converted by its epilogue team and, for a tile's first group, the
        // tile's observations are written.
        __device__ bool group(uint8_t* smem, uint32_t x_base, uint32_t tbase, Bars& b, uint32_t tt,
                              int op, int* err) {
            if (sl.total > 0 && !spin(b, &b.ep_done[S], (sl.total - 1) & 1u, err)) return false;
            if (op == 0 && !spin(b, &b.x_full[tt % NX], (tt / NX) & 1u, err)) return false;
            const uint32_t h = tbase + 256u * S, acc = h + 128u;
            const uint32_t idesc = tc::instr_desc(128, 128, 1);
            tc::fence_after_sync();
            if (op == 0) {
                const int buf = (int)(tt % NX);
#pragma unroll
                for (int j = 0; j < 2; ++j) {
                    uint64_t da = tc::smem_desc(x_base + (uint32_t)buf * kXBytes, kLboX, 128);
                    uint64_t db = tc::smem_desc(smem_u32(smem + kW1) + 2048u * j, kLboW, 128);
#pragma unroll
                    for (int k = 0; k < K1 / 16; ++k) {
                        tc::mma_bf16(j == 0 ? acc : h, da, db, idesc, k != 0);
                        da += (2u * kLboX) >> 4;
                        db += (2u * kLboW) >> 4;
                    }
                }
                tc::mma_commit(&b.acc_full[S]);
                tc::mma_commit(&b.x_free[buf]);                  // X(tt) is no longer read
            } else {
                uint64_t db = tc::smem_desc(smem_u32(smem + kW2) + 2048u * (op - 1), kLboW, 128);
#pragma unroll
                for (int k = 0; k < 16; ++k) {
                    mma_ts(acc, h + h1_col(k), db, idesc, k != 0);
                    db += (2u * kLboW) >> 4;
                }
                tc::mma_commit(&b.acc_full[S]);
            }
            ++sl.total;
            return true;
        }

        __device__ void run(uint8_t* smem, uint32_t x_base, uint32_t tbase, Bars& b, uint32_t n,
                            int* err) {
            const uint32_t end = t + n;
            for (uint32_t tt = t + ((t & 1u) == (uint32_t)S ? 0u : 1u); tt < end; tt += 2)
                for (int op = 0; op < kOps; ++op)
                    if (!group(smem, x_base, tbase, b, tt, op, err)) {
                        t = end;
                        return;
                    }
            t = end;
        }
        // Before the tensor memory is released: every MMA this thread issued
        // has completed.
        __device__ void finish(Bars& b, int* err) {
            tc::mma_commit(&b.drained[S]);
            if (!mbar_wait_bounded(&b.drained[S], 0u, kWaitLimitNs)) atomicOr(err, ERRBIT_TIMEOUT);
            tc::fence_after_sync();
        }
    };

    // --------------------------------------------------------------- epilogue
    // One warp of slot S's epilogue team (S = warp / TW). Warp w of a team
    // handles lane quarter w % 4 and the accumulator columns of its part
    // (w / 4): 64 columns when TW = 8, all 128 (two passes of 64) when TW = 4.
    template <int S>
    struct Epilogue {
        static constexpr int kPasses = 2 / kSplit;            // 64-column passes per group
        uint32_t t = 0;               // first tile of the next run
        Slot sl;
        uint32_t pt = 0;              // partial tiles written (all runs)
        float d[2][4];                // partial logits: [row block][m16n8 accumulator]
        uint32_t w3[2][4][2];         // TW = 8: layer-3 B fragments [L2 half][block][b0, b1]
        uint32_t p_base_off = 0;      // byte offset of the partial buffers in shared memory

        __device__ static int quarter() { return (int)(threadIdx.x >> 5) & 3; }
        __device__ static int part() { return kSplit == 2 ? (int)(threadIdx.x >> 7) & 1 : 0; }

        // Layer-3 B fragment (action g = lane / 4) for the 16 neurons k0 .. k0 + 15.
        __device__ static void w3_frag(const uint8_t* smem, int k0, uint32_t& b0, uint32_t& b1) {
            const int lane = threadIdx.x & 31, g = lane >> 2, tq = lane & 3;
            b0 = *reinterpret_cast<const uint32_t*>(smem + kW3 + tc::cm_offset(g, k0 + 2 * tq, 16, 2));
            b1 = *reinterpret_cast<const uint32_t*>(smem + kW3 + tc::cm_offset(g, k0 + 8 + 2 * tq, 16, 2));
        }

        // TW = 8: loads this warp's W3 fragments into registers (after the
        // policy is staged; again after a restage).
        __device__ void init(const uint8_t* smem) {
            if constexpr (kSplit == 2) {
#pragma unroll
                for (int half = 0; half < 2; ++half)
#pragma unroll
                    for (int kb = 0; kb < 4; ++kb)
                        w3_frag(smem, 128 * half + 64 * part() + 16 * kb, w3[half][kb][0], w3[half][kb][1]);
            }
        }

        // bf16(relu(v + bias)) of 32 columns (lane = row), packed in pairs.
        __device__ static void convert(const uint32_t (&v)[32], const float* bias, uint32_t (&pk)[16]) {
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const float4 bb = *reinterpret_cast<const float4*>(bias + 4 * i);
                pk[2 * i] = tc::bias_relu_bf16x2(__uint_as_float(v[4 * i]), __uint_as_float(v[4 * i + 1]),
                                                 bb.x, bb.y);
                pk[2 * i + 1] = tc::bias_relu_bf16x2(__uint_as_float(v[4 * i + 2]),
                                                     __uint_as_float(v[4 * i + 3]), bb.z, bb.w);
            }
        }

        // Group 0's epilogue: h1 of this warp's columns of H (neurons 128 + c ..)
        // and of ACC (neurons c ..), packed into the columns of H it read
        // (32-neuron block B: h1[128 + 32B ..] at H[32B, +16), h1[32B ..] at
        // H[32B + 16, +16)).
        __device__ void serve_l1(uint8_t* smem, uint32_t tbase, Bars& b) {
            const uint32_t h = tbase + 256u * S, acc = h + 128u;
            const uint32_t lane_q = (uint32_t)(32 * quarter()) << 16;
            const float* b1 = reinterpret_cast<const float*>(smem + kB1);
            tc::fence_after_sync();
            uint32_t v[32], pk[16];
#pragma unroll
            for (int ps = 0; ps < kPasses; ++ps) {
                const uint32_t c0 = 64u * (part() * kPasses + ps);
#pragma unroll
                for (int c = 0; c < 2; ++c) {
                    tc::tmem_ld32x1(h + lane_q + c0 + 32u * c, v);
                    convert(v, b1 + 128 + c0 + 32 * c, pk);
                    tc::tmem_st16(h + lane_q + c0 + 32u * c, pk);
                }
#pragma unroll
                for (int c = 0; c < 2; ++c) {
                    tc::tmem_ld32x1(acc + lane_q + c0 + 32u * c, v);
                    convert(v, b1 + c0 + 32 * c, pk);
                    tc::tmem_st16(h + lane_q + c0 + 32u * c + 16u, pk);
                }
            }
            tc::tmem_wait_st();
            tc::fence_before_sync();
            mbar_arrive_release(&b.ep_done[S]);
        }

        // Group 1 + HALF's epilogue: layer 2's neurons 128 HALF + c .. of the 32
        // rows of this warp's lane quarter (two 16-row blocks), then their share
        // of layer 3 into the partial logits d.
        template <int HALF>
        __device__ void serve_l2(uint8_t* smem, uint32_t tbase, Bars& b, int* err) {
            const int lane = threadIdx.x & 31, g = lane >> 2, tq = lane & 3;
            const uint32_t acc = tbase + 256u * S + 128u;
            const uint32_t lane_q = (uint32_t)(32 * quarter()) << 16;
            tc::fence_after_sync();
            if (HALF == 0) {
#pragma unroll
                for (int rb = 0; rb < 2; ++rb)
#pragma unroll
                    for (int i = 0; i < 4; ++i) d[rb][i] = 0.f;
            }
#pragma unroll
            for (int ps = 0; ps < kPasses; ++ps) {
                const uint32_t c0 = 64u * (part() * kPasses + ps);
                const float* b2 = reinterpret_cast<const float*>(smem + kB2) + 128 * HALF + c0;
#pragma unroll
                for (int rb = 0; rb < 2; ++rb)
#pragma unroll
                    for (int cc = 0; cc < 2; ++cc) {
                        uint32_t x[16];
                        tc::tmem_ld16x256b_x4(acc + lane_q + ((uint32_t)(16 * rb) << 16) + c0 + 32u * cc, x);
                        if (ps == kPasses - 1 && rb == 1 && cc == 1) {
                            tc::fence_before_sync();
                            mbar_arrive_release(&b.ep_done[S]);    // the accumulator is read
                        }
#pragma unroll
                        for (int kh = 0; kh < 2; ++kh) {
                            // 16-neuron block kb of these 64: this thread's columns
                            // 16 kb + 2 tq (+1) and 16 kb + 8 + 2 tq (+1)
                            const int kb = 2 * cc + kh;
                            const float2 bl = *reinterpret_cast<const float2*>(b2 + 16 * kb + 2 * tq);
                            const float2 bh = *reinterpret_cast<const float2*>(b2 + 16 * kb + 8 + 2 * tq);
                            const uint32_t* xx = x + 8 * kh;
                            uint32_t a[4];
                            a[0] = tc::bias_relu_bf16x2(__uint_as_float(xx[0]), __uint_as_float(xx[1]), bl.x, bl.y);
                            a[1] = tc::bias_relu_bf16x2(__uint_as_float(xx[2]), __uint_as_float(xx[3]), bl.x, bl.y);
                            a[2] = tc::bias_relu_bf16x2(__uint_as_float(xx[4]), __uint_as_float(xx[5]), bh.x, bh.y);
                            a[3] = tc::bias_relu_bf16x2(__uint_as_float(xx[6]), __uint_as_float(xx[7]), bh.x, bh.y);
                            uint32_t b0, b1;
                            if constexpr (kSplit == 2) {
                                b0 = w3[HALF][kb][0];
                                b1 = w3[HALF][kb][1];
                            } else {
                                w3_frag(smem, 128 * HALF + (int)c0 + 16 * kb, b0, b1);
                            }
                            mma_m16n8k16(d[rb], a, b0, b1);
                        }
                    }
            }
            if (HALF == 1) {
                // partials of this warp's neurons: rows 32 q + 16 rb + g (+ 8),
                // actions 2 tq, 2 tq + 1
                const uint32_t k = pt++;
                if (k > 0) wait(b, &b.p_free[S], (k - 1) & 1u, err);
                float* pp = reinterpret_cast<float*>(smem + p_base_off + S * kPBytes) + part() * 128 * A;
#pragma unroll
                for (int rb = 0; rb < 2; ++rb)
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        const int row = 32 * quarter() + 16 * rb + g + 8 * (i >> 1);
                        const int a = 2 * tq + (i & 1);
                        if (a < A) pp[row * A + a] = d[rb][i];
                    }
                __syncwarp();
                if (lane == 0) mbar_arrive_release(&b.p_full[S]);
            }
        }

        // Serves every group of the slot's tiles among t .. t + n - 1.
        __device__ void run(uint8_t* smem, uint32_t tbase, Bars& b, uint32_t n, int* err) {
            const uint32_t end = t + n;
            for (uint32_t tt = t + ((t & 1u) == (uint32_t)S ? 0u : 1u); tt < end; tt += 2) {
                wait(b, &b.acc_full[S], sl.total++ & 1u, err);
                serve_l1(smem, tbase, b);
                wait(b, &b.acc_full[S], sl.total++ & 1u, err);
                serve_l2<0>(smem, tbase, b, err);
                wait(b, &b.acc_full[S], sl.total++ & 1u, err);
                serve_l2<1>(smem, tbase, b, err);
            }
            t = end;
        }
    };
};

}  // namespace malib
