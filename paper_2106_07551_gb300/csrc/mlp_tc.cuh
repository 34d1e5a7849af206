// bf16 policy forward on the 5th-generation tensor cores for one tile of 128
// rows (observations of agents that share one policy):
//   logits = W3 relu(W2 relu(W1 x + b1) + b2) + b3
// with bf16 weights and bf16 layer inputs, fp32 accumulation in tensor memory.
//
// Shared memory holds the policy's weight image (staged once by bulk copy):
// W1 [H][K1], W2 [H][H], W3 [NOUT][H] in the core-matrix K-major layout of
// tc_common.cuh (K1 = input width padded to 16, NOUT = actions padded to 16),
// then the fp32 biases b1 [H], b2 [H], b3 [NOUT] (staged with the image or read
// from global memory). The caller's observation tile X [128][K1] (same layout)
// is layer 1's A operand; the hidden activations never touch shared memory:
// each layer's epilogue reads its fp32 accumulator from tensor memory, applies
// ReLU, rounds to bf16 and writes the packed result back to tensor memory,
// where the next layer's MMAs read it as their A operand (two bf16 per
// 32-bit column, the lower k in the low half, row i in lane i).
//
// Tensor-memory columns (512 allocated):
//   D1  [0, 256)    layer-1 accumulator
//   H1  [256, 384)  h1, packed
//   D2a [384, 512)  layer-2 accumulator, outputs 0..127
//   D2b [0, 128)    layer-2 accumulator, outputs 128..255 (D1's first half)
//   H2  [128, 256)  h2, packed (D1's second half)
//   D3  [384, 448)  layer 3 as four 16-column partial sums (D2a's first part)
// Each layer's epilogue runs in two column halves. Layer 2's MMAs over h1's
// first half are issued as soon as it is written, and layer 2 is split by
// output halves so that the first half's epilogue starts while the tensor core
// computes the second; layer 3 likewise follows h2's halves. Thread 0 issues
// the MMAs; the engine's 8 warps split each epilogue (warp w: TMEM lane
// quarter w % 4, 64 of the 128 columns of a half), which adds the layer's bias
// (one packed add per pair of values) before ReLU and rounding.
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
    static constexpr uint32_t kSmemBytes = kStageBytes;             // the engine's shared memory
    static_assert(kStageBytes % 16 == 0, "16-byte aligned image");
    static constexpr uint32_t kXBytes = 128 * K1 * 2;               // one observation tile
    static constexpr uint32_t kTmemCols = 512;
    static constexpr int kD1 = 0, kH1 = 256, kD2a = 384, kD2b = 0, kH2 = 128, kD3 = 384;
    static constexpr uint32_t kLboX = (128 / 8) * 128;              // K-chunk stride, 128 rows
    static constexpr uint32_t kLboW = (H / 8) * 128;                // K-chunk stride, H rows
    static constexpr uint32_t kLboW3 = (NOUT / 8) * 128;

    // Byte offset, inside an observation tile, of the 8 bf16 columns k..k+7 of row.
    __device__ static uint32_t x_offset(int row, int k) { return tc::cm_offset(row, k, 128, 2); }

    // Barrier over the engine's threads.
    __device__ static void sync() {
        if (kBarId == 0) {
            __syncthreads();
        } else {
            asm volatile("bar.sync %0, 256;" ::"n"(kBarId) : "memory");
        }
    }

    // Orders this thread's tensor-memory stores (and loads) before the next
    // MMA, through a barrier of the engine's threads (all engine threads call).
    __device__ static void handoff() {
        tc::tmem_wait_st();
        tc::fence_before_sync();
        sync();
        tc::fence_after_sync();
    }

    // Waits (bounded) for the current phase of MMA barrier i (bars[i]); bit i
    // of `parity` tracks that barrier's phase and is flipped. Two barriers: the
    // two halves of layer 2 complete back to back, and a thread that looked late
    // at one barrier whose next phase had already completed would miss it.
    __device__ static void wait_mma(uint64_t* bars, int i, uint32_t& parity, int* err) {
        if (!mbar_wait_bounded(bars + i, (parity >> i) & 1u, kWaitLimitNs) && threadIdx.x == 0)
            atomicOr(err, ERRBIT_TIMEOUT);
        parity ^= 1u << i;
        tc::fence_after_sync();
    }

    // tcgen05.mma kind::f16 with the A operand in tensor memory.
    __device__ static void mma_ta(uint32_t d_tmem, uint32_t a_tmem, uint64_t b, uint32_t idesc,
                                  bool accumulate) {
        asm volatile(
            "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
            " tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n}" ::"r"(d_tmem),
            "r"(a_tmem), "l"(b), "r"(idesc), "r"((uint32_t)accumulate)
            : "memory");
    }

    // Issued by thread 0: D (+)= A(tensor memory, K steps [s0, s1), 8 columns
    // per step from a_col) . B^T, B from the weight image at w (K-chunk stride
    // lbo_w). Consecutive K steps advance the descriptor's start-address field
    // (bits 0-13, address >> 4) by a constant; shared-memory addresses stay
    // below 2^18, so the field never carries.
    __device__ static void issue_ta(uint32_t d, uint32_t a_col, uint32_t w, uint32_t lbo_w, int s0,
                                    int s1, uint32_t idesc, bool accumulate_first) {
        uint64_t db = tc::smem_desc(w + 2u * s0 * lbo_w, lbo_w, 128);
        for (int s = s0; s < s1; ++s) {
            mma_ta(d, a_col + 8u * s, db, idesc, accumulate_first || s != s0);
            db += (2u * lbo_w) >> 4;
        }
    }

    // One 32-column chunk of an accumulator (in registers) -> relu -> bf16 pairs
    // -> 16 packed tensor-memory columns at taddr. With `bias`, the chunk's 32
    // bias values are added first.
    __device__ static void pack_chunk(const uint32_t (&v)[32], const float* bias, uint32_t taddr) {
        uint32_t pk[16];
        if (bias) {
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const float4 b = kSmemBias ? *reinterpret_cast<const float4*>(bias + 4 * j)
                                           : __ldg(reinterpret_cast<const float4*>(bias + 4 * j));
                pk[2 * j] = tc::bias_relu_bf16x2(__uint_as_float(v[4 * j]),
                                                 __uint_as_float(v[4 * j + 1]), b.x, b.y);
                pk[2 * j + 1] = tc::bias_relu_bf16x2(__uint_as_float(v[4 * j + 2]),
                                                     __uint_as_float(v[4 * j + 3]), b.z, b.w);
            }
        } else {
#pragma unroll
            for (int j = 0; j < 16; ++j)
                pk[j] = tc::relu_bf16x2(__uint_as_float(v[2 * j]), __uint_as_float(v[2 * j + 1]));
        }
        tc::tmem_st16(taddr, pk);
    }

    // One 128-column half of a layer's output: accumulator columns
    // [dcol, dcol + 128) plus bias -> packed activations at [hcol, hcol + 64).
    // Warp w takes lane quarter w % 4 and columns 64 (w / 4) .. of the half;
    // bias covers the half's columns.
    __device__ static void epilogue_half(uint32_t tbase, int dcol, int hcol, const float* bias) {
        const int warp = threadIdx.x >> 5;
        const int q = warp & 3, h = warp >> 2;
        const int c = 64 * h;
        uint32_t r0[32], r1[32];
        tc::tmem_ld32x2(tc::tmem_addr(tbase, 32 * q, dcol + c), tc::tmem_addr(tbase, 32 * q, dcol + c + 32),
                        r0, r1);
        pack_chunk(r0, bias ? bias + c : nullptr, tc::tmem_addr(tbase, 32 * q, hcol + c / 2));
        pack_chunk(r1, bias ? bias + c + 32 : nullptr, tc::tmem_addr(tbase, 32 * q, hcol + c / 2 + 16));
    }

    // The helper's part of a forward given h1_ready, called by one thread after
    // the phase of h1_ready[part] (and tcgen05-fenced after it), in order: part 0
    // (h1's first half stored) issues layer 2's outputs 0..127 over it; part 1
    // (all of h1 stored) the rest of those outputs, committed on bars[0], then
    // outputs 128..255 into D2b over all of h1, committed on bars[1]. One
    // thread issues every layer-2 MMA, so they execute in order.
    // (Issuing layer 3 from the helper as well was slower: it sits on the
    // forward's critical path, where the helper's response time shows.)
    // The helper's part of a forward when only layer 2's second output half is
    // delegated (helper_all false): after the phase of h1_ready[0], outputs
    // 128..255 into D2b over all of h1, committed on bars[1].
    __device__ static void issue_layer2b(const uint8_t* smem, uint32_t tbase, uint64_t* bars) {
        issue_ta(tbase + kD2b, tbase + kH1, smem_u32(smem + kW2) + (H / 2 / 8) * 128, kLboW, 0, H / 16,
                 tc::instr_desc(128, H / 2, 1), false);
        tc::mma_commit(bars + 1);
    }

    __device__ static void issue_layer2(const uint8_t* smem, uint32_t tbase, uint64_t* bars, int part) {
        const uint32_t s_w2 = smem_u32(smem + kW2), idesc_half = tc::instr_desc(128, H / 2, 1);
        constexpr int kS = H / 16;
        if (part == 0) {
            issue_ta(tbase + kD2a, tbase + kH1, s_w2, kLboW, 0, kS / 2, idesc_half, false);
            return;
        }
        issue_ta(tbase + kD2a, tbase + kH1, s_w2, kLboW, kS / 2, kS, idesc_half, true);
        tc::mma_commit(bars);                               // D2a complete
        issue_ta(tbase + kD2b, tbase + kH1, s_w2 + (H / 2 / 8) * 128, kLboW, 0, kS, idesc_half, false);
        tc::mma_commit(bars + 1);                           // D2b complete
    }

    // Full forward of the 128-row observation tile at shared-memory address
    // x_tile. bars: two mbarriers (count 1) for the MMA completions; parity:
    // their phase bits, kept by the caller across forwards. out(row, logits[16]) is called by the threads of warps 0-3 (thread
    // = row) for every row; the caller knows which rows hold observations.
    // gbias: the policy's biases in global memory (used when kSmemBias is false).
    // All engine threads call.
    // x_published: the caller's X writers already fenced (proxy) and the engine
    // has synchronised since, so MMA 1 issues at once; otherwise the forward
    // fences and synchronises first.
    template <class Out>
    // h1_ready (optional, two mbarriers of count 1): part of layer 2 is issued
    // by another, otherwise idle thread, so that thread 0's warp is not held
    // while the tensor core retires those MMAs. helper_all false: thread 0
    // issues outputs 0..127 and arrives on h1_ready[0] once h1 is complete;
    // the helper issues outputs 128..255 (issue_layer2b). helper_all true:
    // thread 0 arrives on h1_ready[0] when h1's first half is stored and on
    // h1_ready[1] when all of h1 is; the helper issues all of layer 2
    // (issue_layer2). Two barriers, because both arrivals may land before the
    // helper looks: on one barrier the second would return its phase parity to
    // the value the helper waits for. No barrier can run a phase ahead, since
    // the next forward needs this one's layer 2.
    // w2_ready (optional, with its phase parity): an mbarrier whose phase
    // completes when W2 and W3 have landed in shared memory; thread 0 waits
    // on it (bounded) before the first layer-2 MMA, so that a restage of
    // those weights overlaps layer 1 and its epilogue.
    __device__ static void forward(uint8_t* smem, const float* gbias, uint32_t tbase, uint64_t* bars,
                                   uint32_t& parity, int* err, Out out, uint32_t x_tile,
                                   bool x_published = false, uint64_t* h1_ready = nullptr,
                                   uint64_t* w2_ready = nullptr, uint32_t w2_parity = 0,
                                   bool helper_all = false) {
        uint64_t* const h1_all = helper_all ? h1_ready : nullptr;   // the helper issues all of layer 2
        const float* bias = kSmemBias ? reinterpret_cast<const float*>(smem + kBias) : gbias;
        const uint32_t s_w1 = smem_u32(smem + kW1), s_w2 = smem_u32(smem + kW2);
        const uint32_t s_w3 = smem_u32(smem + kW3);
        if (!x_published) {
            fence_proxy_async_smem();
            tc::fence_before_sync();
            sync();
        }
        if (threadIdx.x == 0) fence_proxy_async_smem();
        tc::fence_after_sync();
        const uint32_t idesc_full = tc::instr_desc(128, H, 1);
        const uint32_t idesc_half = tc::instr_desc(128, H / 2, 1);
        const uint32_t idesc3 = tc::instr_desc(128, NOUT, 1);
        constexpr int kS = H / 16;                      // K steps of layers 2 and 3
        // layer 1 (N = 256, K = K1) into D1
        if (threadIdx.x == 0) {
            uint64_t da = tc::smem_desc(x_tile, kLboX, 128);
            uint64_t db = tc::smem_desc(s_w1, kLboW, 128);
            for (int s = 0; s < K1 / 16; ++s) {
                tc::mma_bf16(tbase + kD1, da, db, idesc_full, s != 0);
                da += (2u * kLboX) >> 4;
                db += (2u * kLboW) >> 4;
            }
            tc::mma_commit(bars);
        }
        wait_mma(bars, 0, parity, err);
        // h1, first half; then layer 2's outputs 0..127 over h1's first half
        epilogue_half(tbase, kD1, kH1, bias);
        handoff();
        if (threadIdx.x == 0) {
            // the W2 wait comes first: with a helper, its acquire reaches the
            // helper through the release of the arrival below
            if (w2_ready && !mbar_wait_bounded(w2_ready, w2_parity, kWaitLimitNs))
                atomicOr(err, ERRBIT_TIMEOUT);
            if (h1_all) {
                tc::fence_before_sync();
                mbar_arrive_release(h1_all);                // part 0 is issued by the helper
            } else {
                issue_ta(tbase + kD2a, tbase + kH1, s_w2, kLboW, 0, kS / 2, idesc_half, false);
            }
        }
        // h1, second half; then the rest of layer 2: outputs 0..127, then
        // 128..255 into D2b (D1's first half, already read)
        epilogue_half(tbase, kD1 + H / 2, kH1 + H / 4, bias + H / 2);
        handoff();
        if (threadIdx.x == 0) {
            if (h1_all) {
                tc::fence_before_sync();
                mbar_arrive_release(h1_all + 1);            // part 1 is issued by the helper
            } else {
                issue_ta(tbase + kD2a, tbase + kH1, s_w2, kLboW, kS / 2, kS, idesc_half, true);
                tc::mma_commit(bars);                       // D2a complete
                if (h1_ready) {
                    tc::fence_before_sync();
                    mbar_arrive_release(h1_ready);          // D2b is issued by the helper
                } else {
                    issue_ta(tbase + kD2b, tbase + kH1, s_w2 + (H / 2 / 8) * 128, kLboW, 0, kS,
                             idesc_half, false);
                    tc::mma_commit(bars + 1);               // D2b complete
                }
            }
        }
        wait_mma(bars, 0, parity, err);                     // D2a
        // h2, first half (into H2, D1's second half, already read); then layer 3
        // over it: four chains of 4 K steps into D3 (D2a's columns, just read)
        epilogue_half(tbase, kD2a, kH2, bias + H);
        handoff();
        auto mma3 = [&](int s0, int s1) {
            uint64_t db = tc::smem_desc(s_w3 + 2u * s0 * kLboW3, kLboW3, 128);
            for (int s = s0; s < s1; ++s) {
                mma_ta(tbase + kD3 + (uint32_t)(16 * (s / (kS / 4))), tbase + kH2 + 8u * s, db,
                       idesc3, (s % (kS / 4)) != 0);
                db += (2u * kLboW3) >> 4;
            }
        };
        if (threadIdx.x == 0) mma3(0, kS / 2);
        wait_mma(bars, 1, parity, err);                     // D2b
        epilogue_half(tbase, kD2b, kH2 + H / 4, bias + H + H / 2);
        handoff();
        if (threadIdx.x == 0) {
            mma3(kS / 2, kS);
            tc::mma_commit(bars);
        }
        wait_mma(bars, 0, parity, err);
        const int warp = threadIdx.x >> 5;
        if (warp < 4) {
            const int row = threadIdx.x;
            float v[16];
            {
                uint32_t r[32], r2[32];
                tc::tmem_ld32x2(tc::tmem_addr(tbase, 32 * warp, kD3),
                                tc::tmem_addr(tbase, 32 * warp, kD3 + 32), r, r2);
#pragma unroll
                for (int i = 0; i < 16; ++i)
                    v[i] = (__uint_as_float(r[i]) + __uint_as_float(r[16 + i])) +
                           (__uint_as_float(r2[i]) + __uint_as_float(r2[16 + i]));
            }
#pragma unroll
            for (int i = 0; i < 16; ++i) v[i] += kSmemBias ? bias[2 * H + i] : __ldg(bias + 2 * H + i);
            out(row, v);
        }
        // the next forward's MMAs overwrite D1, D2b and H2's columns: every
        // tensor-memory load of this one is complete before the barrier
        tc::fence_before_sync();
        sync();
    }
};

}  // namespace malib
