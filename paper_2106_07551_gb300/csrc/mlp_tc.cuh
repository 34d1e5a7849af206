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
// layer's output, so X, h1 and h2 reuse the same 64 KB. One 256-column TMEM
// accumulator is
// reused by the three layers. Thread 0 issues the MMAs; the 8 warps split each
// epilogue (warp w: TMEM lane quarter w % 4, column half w / 4).
#pragma once

#include <cstdint>

#include "device_common.cuh"
#include "tc_common.cuh"

namespace malib {

// kSmemBias: stage the biases with the weights (true) or read them from the
// policy's global image through L1 (false, when shared memory is short).
template <int K1, int H, int NOUT, bool kSmemBias = true>
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
    static constexpr uint32_t kTmemCols = 256;
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

    // Issued by thread 0: D(tmem) = A(act tile, K) . B^T (B: n_rows x K image).
    __device__ static void issue(uint32_t tbase, uint32_t act, uint32_t w, uint32_t lbo_w, int K,
                                 uint32_t idesc) {
        for (int s = 0; s < K / 16; ++s)
            tc::mma_bf16(tbase, tc::smem_desc(act + 2u * s * kLboAct, kLboAct, 128),
                         tc::smem_desc(w + 2u * s * lbo_w, lbo_w, 128), idesc, s > 0);
    }

    // D + bias -> relu -> bf16 into the activation tile (this thread: one row,
    // one half of the H columns, in 32-column chunks; the next chunk's tensor
    // memory load and bias loads are in flight while the current chunk is
    // processed).
    __device__ static void epilogue_hidden(uint8_t* act, const float* bias, uint32_t tbase) {
        const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
        const int q = warp & 3, half = warp >> 2;
        const int row = 32 * q + lane;
        constexpr int kChunks = H / 2 / 32;
        uint32_t r[2][32];
        float4 bs[2][8];
        auto load_bias = [&](int buf, int c0) {
#pragma unroll
            for (int j = 0; j < 8; ++j)
                bs[buf][j] = kSmemBias ? *reinterpret_cast<const float4*>(bias + c0 + 4 * j)
                                       : __ldg(reinterpret_cast<const float4*>(bias + c0 + 4 * j));
        };
        tc::tmem_ld32_nowait(tc::tmem_addr(tbase, 32 * q, half * (H / 2)), r[0]);
        load_bias(0, half * (H / 2));
        tc::tmem_wait_ld();
#pragma unroll
        for (int cc = 0; cc < kChunks; ++cc) {
            const int c0 = half * (H / 2) + cc * 32;
            if (cc + 1 < kChunks) {
                tc::tmem_ld32_nowait(tc::tmem_addr(tbase, 32 * q, c0 + 32), r[(cc + 1) & 1]);
                load_bias((cc + 1) & 1, c0 + 32);
            }
            const uint32_t* v = r[cc & 1];
            const float4* b = bs[cc & 1];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const float4 b0 = b[2 * j], b1 = b[2 * j + 1];
                uint4 pk;
                pk.x = tc::pack_bf16(fmaxf(__uint_as_float(v[8 * j + 0]) + b0.x, 0.f),
                                     fmaxf(__uint_as_float(v[8 * j + 1]) + b0.y, 0.f));
                pk.y = tc::pack_bf16(fmaxf(__uint_as_float(v[8 * j + 2]) + b0.z, 0.f),
                                     fmaxf(__uint_as_float(v[8 * j + 3]) + b0.w, 0.f));
                pk.z = tc::pack_bf16(fmaxf(__uint_as_float(v[8 * j + 4]) + b1.x, 0.f),
                                     fmaxf(__uint_as_float(v[8 * j + 5]) + b1.y, 0.f));
                pk.w = tc::pack_bf16(fmaxf(__uint_as_float(v[8 * j + 6]) + b1.z, 0.f),
                                     fmaxf(__uint_as_float(v[8 * j + 7]) + b1.w, 0.f));
                *reinterpret_cast<uint4*>(act + act_offset(row, c0 + 8 * j)) = pk;
            }
            if (cc + 1 < kChunks) tc::tmem_wait_ld();
        }
    }

    // Makes this CTA's generic shared-memory writes visible to the tensor cores
    // and orders tensor-memory reads before the next MMA (all threads call).
    __device__ static void handoff() {
        fence_proxy_async_smem();
        tc::fence_before_sync();
        __syncthreads();
        tc::fence_after_sync();
    }

    // Full forward of the 128-row tile whose X has been written (and published
    // by the caller's synchronisation). out(row, logits[16]) is called by the
    // threads of warps 0-3 (thread = row) for every row; the caller knows which
    // rows hold observations. gbias: the policy's biases in global memory (used
    // when kSmemBias is false). All threads call.
    // x_published: the caller's X writers already fenced (proxy) and the CTA
    // has synchronised since (e.g. a cluster sync), so MMA 1 issues at once.
    template <class Out>
    __device__ static void forward(uint8_t* smem, const float* gbias, uint32_t tbase, uint64_t* bar,
                                   uint32_t& parity, int* err, Out out, bool x_published = false) {
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
        if (threadIdx.x == 0) {
            issue(tbase, s_act, s_w1, kLboW, K1, tc::instr_desc(128, H, 1));
            tc::mma_commit(bar);
        }
        wait_mma(bar, parity, err);
        epilogue_hidden(act, bias, tbase);
        handoff();
        if (threadIdx.x == 0) {
            issue(tbase, s_act, s_w2, kLboW, H, tc::instr_desc(128, H, 1));
            tc::mma_commit(bar);
        }
        wait_mma(bar, parity, err);
        epilogue_hidden(act, bias + H, tbase);
        handoff();
        if (threadIdx.x == 0) {
            // four independent accumulators (TMEM columns 16j..16j+15) over K
            // quarters, so the 16 small MMAs form 4 short chains
            const uint32_t idesc3 = tc::instr_desc(128, NOUT, 1);
            for (int s = 0; s < H / 16; ++s)
                tc::mma_bf16(tbase + (uint32_t)(16 * (s / (H / 64))),
                             tc::smem_desc(s_act + 2u * s * kLboAct, kLboAct, 128),
                             tc::smem_desc(s_w3 + 2u * s * kLboW3, kLboW3, 128), idesc3,
                             (s % (H / 64)) != 0);
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
        tc::fence_before_sync();
        __syncthreads();
    }
};

}  // namespace malib
