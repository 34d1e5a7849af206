// bf16 policy forward on the 5th-generation tensor cores for one tile of 128
// rows (observations of agents that share one policy):
//   logits = W3 relu(W2 relu(W1 x + b1) + b2) + b3
// with bf16 weights and bf16 layer inputs, fp32 accumulation in tensor memory.
//
// Shared memory holds the policy's weight image (staged once by bulk copy):
// W1 [H][K1], W2 [H][H], W3 [NOUT][H] in the core-matrix K-major layout of
// tc_common.cuh (K1 = input width padded to 16, NOUT = actions padded to 16),
// then the fp32 biases b1 [H], b2 [H], b3 [NOUT] (staged with the image), then
// one activation tile [128][H]. The observation tile X [128][K1] lives at the
// start of that activation tile: every layer's A operand is the previous
// layer's output, so X, h1 and h2 reuse the same 64 KB. Tensor memory holds
// two 256-column accumulators: layer 1 writes D1 (columns 0..255), layer 2 D2
// (256..511), layer 3 four 16-column partial sums over D1's first 64 columns.
// D1 and D2 start each forward holding their layer's bias (written with
// tcgen05.st while other work waits: b2 during layer 1's MMA, b1 after the
// previous forward), so the MMAs accumulate onto it and the epilogues only
// apply ReLU and bf16 rounding. Thread 0 issues the MMAs; the 8 warps split
// each epilogue (warp w: TMEM lane quarter w % 4, 64 of the 128 columns of a
// half). Each layer's epilogue runs in two column halves, and the next layer's
// MMAs over the first half's K range are issued before the second half is
// produced, so the tensor core works while the epilogue warps drain tensor
// memory.
#pragma once

#include <cstdint>

#include "device_common.cuh"
#include "tc_common.cuh"

namespace malib {

// kSmemBias: stage the biases with the weights (true) or read them from the
// policy's global image through L1 (false, when shared memory is short).
// kBarId: 0 - the whole CTA runs the engine (CTA barriers); otherwise the
// engine runs on warps 0-7 alone and synchronises them with named barrier
// kBarId (256 threads), leaving the CTA's other warps free for other work.
template <int K1, int H, int NOUT, bool kSmemBias = true, int kBarId = 0>
struct MlpTc {
    static_assert(K1 % 16 == 0 && H == 256 && NOUT == 16, "shapes built: K1 % 16, H 256, NOUT 16");
    static constexpr uint32_t kW1 = 0;
    static constexpr uint32_t kW2 = kW1 + H * K1 * 2;
    static constexpr uint32_t kW3 = kW2 + H * H * 2;
    static constexpr uint32_t kImageBytes = kW3 + NOUT * H * 2;     // staged into shared memory
    static constexpr uint32_t kBiasFloats = H + H + NOUT;           // b1, b2, b3 after the image
    static constexpr uint32_t kPolicyBytes = kImageBytes + kBiasFloats * 4;   // global image
    static constexpr uint32_t kStageBytes = kSmemBias ? kPolicyBytes : kImageBytes;
    static constexpr uint32_t kBias = kImageBytes;                  // biases (after the image)
    static constexpr uint32_t kAct = kStageBytes;                   // activation tile offset
    static constexpr uint32_t kActBytes = 128 * H * 2;
    static constexpr uint32_t kSmemBytes = kStageBytes + kActBytes;
    static_assert(kStageBytes % 16 == 0, "activation tile 16-byte aligned");
    static constexpr uint32_t kTmemCols = 512;    // D1 [0,256), D2 [256,512), D3 [0,64)
    static constexpr uint32_t kLboAct = (128 / 8) * 128;            // K-chunk stride, 128 rows
    static constexpr uint32_t kLboW = (H / 8) * 128;                // K-chunk stride, H rows
    static constexpr uint32_t kLboW3 = (NOUT / 8) * 128;

    // Byte offset, inside the activation tile, of the 8 bf16 columns k..k+7 of row.
    __device__ static uint32_t act_offset(int row, int k) { return tc::cm_offset(row, k, 128, 2); }

    // Waits for the MMA barrier's current phase (bounded); flips the parity.
    __device__ static void wait_mma(uint64_t* bar, uint32_t& parity, int* err) {
        if (!mbar_wait_bounded(bar, parity, kWaitLimitNs) && threadIdx.x == 0)
            atomicOr(err, ERRBIT_TIMEOUT);
        parity ^= 1u;
        tc::fence_after_sync();
    }

    // Issued by thread 0: D(tmem) (+)= A(act tile, K steps [s0, s1)) . B^T, where
    // B starts `w` (a row-group offset inside an image whose K-chunk stride is
    // lbo_w). The first step overwrites D when `fresh`.
    // Consecutive K steps advance the descriptors' start-address field (bits
    // 0-13, address >> 4) by a constant; shared-memory addresses stay below
    // 2^18, so the field never carries.
    __device__ static void issue(uint32_t d, uint32_t act, uint32_t w, uint32_t lbo_w, int s0,
                                 int s1, uint32_t idesc, bool fresh) {
        uint64_t da = tc::smem_desc(act + 2u * s0 * kLboAct, kLboAct, 128);
        uint64_t db = tc::smem_desc(w + 2u * s0 * lbo_w, lbo_w, 128);
        const uint64_t step_a = (2u * kLboAct) >> 4, step_b = (2u * lbo_w) >> 4;
        for (int s = s0; s < s1; ++s) {
            tc::mma_bf16(d, da, db, idesc, !(fresh && s == s0));
            da += step_a;
            db += step_b;
        }
    }

    // One 32-column chunk of a layer's output for this thread's row: D (already
    // in registers, bias included) -> relu -> bf16, stored into the activation tile.
    __device__ static void store_chunk(uint8_t* act, int row, int c0, const uint32_t (&v)[32]) {
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            auto f = [&](int i) { return __uint_as_float(v[8 * j + i]); };
            uint4 pk;
            pk.x = tc::relu_bf16x2(f(0), f(1));
            pk.y = tc::relu_bf16x2(f(2), f(3));
            pk.z = tc::relu_bf16x2(f(4), f(5));
            pk.w = tc::relu_bf16x2(f(6), f(7));
            *reinterpret_cast<uint4*>(act + act_offset(row, c0 + 8 * j)) = pk;
        }
    }

    // Writes a layer's bias (H values) into every row of the accumulator at TMEM
    // column tcol, so the layer's MMAs accumulate onto it: warp w writes its lane
    // quarter w % 4, columns 128 (w / 4) .. +127. Waits for its stores.
    __device__ static void prefill(const float* bias, uint32_t tbase, int tcol) {
        const int warp = threadIdx.x >> 5;
        const int q = warp & 3, h = warp >> 2;
#pragma unroll 1
        for (int c = 0; c < 4; ++c) {
            const int c0 = 128 * h + 32 * c;
            uint32_t r[32];
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const float4 b = kSmemBias ? *reinterpret_cast<const float4*>(bias + c0 + 4 * j)
                                           : __ldg(reinterpret_cast<const float4*>(bias + c0 + 4 * j));
                r[4 * j] = __float_as_uint(b.x);
                r[4 * j + 1] = __float_as_uint(b.y);
                r[4 * j + 2] = __float_as_uint(b.z);
                r[4 * j + 3] = __float_as_uint(b.w);
            }
            tc::tmem_st32(tc::tmem_addr(tbase, 32 * q, tcol + c0), r);
        }
        tc::tmem_wait_st();
    }

    // Layer 1's bias into D1 before the first forward of a policy (after its
    // weights and biases are staged). The caller orders it before the next MMA
    // (tcgen05 fence before a barrier of the engine's threads).
    __device__ static void prefill_d1(uint8_t* smem, const float* gbias, uint32_t tbase) {
        prefill(kSmemBias ? reinterpret_cast<const float*>(smem + kBias) : gbias, tbase, 0);
    }

    // A layer's output, D (TMEM columns tcol .., bias included) -> relu -> bf16
    // into the activation tile, in two column halves. Warp w takes TMEM lane quarter
    // w % 4 and, in each half, the 64 columns 64 (w / 4) .. of that half. The
    // first half is stored, then the second half's tensor-memory loads are
    // issued and stay in flight across mid() (the hand-off that lets the next
    // layer's MMAs start on the first half).
    template <class Mid>
    __device__ static void epilogue_layer(uint8_t* act, uint32_t tbase, int tcol, Mid mid) {
        const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
        const int q = warp & 3, h = warp >> 2;
        const int row = 32 * q + lane;
        const int ca = 64 * h, cb = H / 2 + 64 * h;
        {
            uint32_t r0[32], r1[32];
            tc::tmem_ld32_nowait(tc::tmem_addr(tbase, 32 * q, tcol + ca), r0);
            tc::tmem_ld32_nowait(tc::tmem_addr(tbase, 32 * q, tcol + ca + 32), r1);
            tc::tmem_wait_ld();
            store_chunk(act, row, ca, r0);
            store_chunk(act, row, ca + 32, r1);
        }
        uint32_t r2[32], r3[32];
        tc::tmem_ld32_nowait(tc::tmem_addr(tbase, 32 * q, tcol + cb), r2);
        tc::tmem_ld32_nowait(tc::tmem_addr(tbase, 32 * q, tcol + cb + 32), r3);
        mid();
        tc::tmem_wait_ld();
        store_chunk(act, row, cb, r2);
        store_chunk(act, row, cb + 32, r3);
    }

    // Barrier over the engine's threads.
    __device__ static void sync() {
        if (kBarId == 0) {
            __syncthreads();
        } else {
            asm volatile("bar.sync %0, 256;" ::"n"(kBarId) : "memory");
        }
    }

    // Makes the engine's generic shared-memory writes visible to the tensor
    // cores and orders tensor-memory reads before the next MMA (all engine
    // threads call).
    __device__ static void handoff() {
        fence_proxy_async_smem();
        tc::fence_before_sync();
        sync();
        tc::fence_after_sync();
    }

    // Full forward of the 128-row tile whose X has been written (and published
    // by the caller's synchronisation). out(row, logits[16]) is called by the
    // threads of warps 0-3 (thread = row) for every row; the caller knows which
    // rows hold observations. gbias: the policy's biases in global memory (used
    // when kSmemBias is false). All threads call.
    // x_published: the caller's X writers already fenced (proxy) and the CTA
    // has synchronised since (e.g. a cluster sync), so MMA 1 issues at once.
    // x_tile: shared-memory address of the observation tile [128][K1] (same
    // core-matrix layout as the activation tile); 0 = the activation tile's start.
    template <class Out>
    __device__ static void forward(uint8_t* smem, const float* gbias, uint32_t tbase, uint64_t* bar,
                                   uint32_t& parity, int* err, Out out, bool x_published = false,
                                   uint32_t x_tile = 0) {
        uint8_t* act = smem + kAct;
        const float* bias = kSmemBias ? reinterpret_cast<const float*>(smem + kBias) : gbias;
        const uint32_t s_act = smem_u32(act);
        const uint32_t s_w1 = smem_u32(smem + kW1), s_w2 = smem_u32(smem + kW2);
        const uint32_t s_w3 = smem_u32(smem + kW3);
        if (x_published) {
            if (threadIdx.x == 0) fence_proxy_async_smem();
            tc::fence_after_sync();
        } else {
            handoff();
        }
        const uint32_t idesc_full = tc::instr_desc(128, H, 1);
        const uint32_t idesc3 = tc::instr_desc(128, NOUT, 1);
        const uint32_t d1 = tbase, d2 = tbase + 256;
        constexpr int kS = H / 16;                      // K steps of layers 2 and 3
        // layer 1 (N = 256, K = K1) onto D1 (holding b1); meanwhile b2 goes into D2
        if (threadIdx.x == 0) {
            issue(d1, x_tile ? x_tile : s_act, s_w1, kLboW, 0, K1 / 16, idesc_full, false);
            tc::mma_commit(bar);
        }
        prefill(bias + H, tbase, 256);
        wait_mma(bar, parity, err);
        // h1 columns 0..127, then layer-2 K steps 0..7 (N = 256) while h1
        // columns 128..255 are produced, then K steps 8..15
        epilogue_layer(act, tbase, 0, [&] {
            handoff();
            if (threadIdx.x == 0) issue(d2, s_act, s_w2, kLboW, 0, kS / 2, idesc_full, false);
        });
        handoff();
        if (threadIdx.x == 0) {
            issue(d2, s_act, s_w2, kLboW, kS / 2, kS, idesc_full, false);
            tc::mma_commit(bar);
        }
        wait_mma(bar, parity, err);
        // h2 columns 0..127, then layer-3 K steps 0..7 while h2 columns
        // 128..255 are produced. Layer 3 runs as 4 chains of 4 MMAs into TMEM
        // columns 16j (D1's columns, free once h1 is written).
        auto mma3 = [&](int s0, int s1) {
            uint64_t da = tc::smem_desc(s_act + 2u * s0 * kLboAct, kLboAct, 128);
            uint64_t db = tc::smem_desc(s_w3 + 2u * s0 * kLboW3, kLboW3, 128);
            for (int s = s0; s < s1; ++s) {
                tc::mma_bf16(tbase + (uint32_t)(16 * (s / (kS / 4))), da, db, idesc3,
                             (s % (kS / 4)) != 0);
                da += (2u * kLboAct) >> 4;
                db += (2u * kLboW3) >> 4;
            }
        };
        epilogue_layer(act, tbase, 256, [&] {
            handoff();
            if (threadIdx.x == 0) mma3(0, kS / 2);
        });
        handoff();
        if (threadIdx.x == 0) {
            mma3(kS / 2, kS);
            tc::mma_commit(bar);
        }
        wait_mma(bar, parity, err);
        const int warp = threadIdx.x >> 5;
        if (warp < 4) {
            const int row = threadIdx.x;
            float v[16];
            {
                uint32_t r[32], r2[32];
                tc::tmem_ld32_nowait(tc::tmem_addr(tbase, 32 * warp, 0), r);
                tc::tmem_ld32_nowait(tc::tmem_addr(tbase, 32 * warp, 32), r2);
                tc::tmem_wait_ld();
#pragma unroll
                for (int i = 0; i < 16; ++i)
                    v[i] = (__uint_as_float(r[i]) + __uint_as_float(r[16 + i])) +
                           (__uint_as_float(r2[i]) + __uint_as_float(r2[16 + i]));
            }
#pragma unroll
            for (int i = 0; i < 16; ++i) v[i] += kSmemBias ? bias[2 * H + i] : __ldg(bias + 2 * H + i);
            out(row, v);
        }
        // b1 into D1 for the next forward (each warp rewrites only columns of its
        // own lane quarter, after its own reads of the layer-3 chains)
        prefill(bias, tbase, 0);
        tc::fence_before_sync();
        sync();
    }
};

}  // namespace malib
