// 5th-generation tensor-core (tcgen05) building blocks for sm_103a: tensor
// memory allocation, shared-memory matrix descriptors in the no-swizzle
// K-major layout, instruction descriptors, MMA issue and completion, and tensor
// memory loads. Single-CTA (cta_group::1) forms only.
//
// Operand layout ("core-matrix K-major, no swizzle"): a tile of R rows x K
// elements is stored as core matrices of 8 rows x 16 bytes (rows 16 bytes
// apart, 128 contiguous bytes). Core matrix (row group g = row / 8, K chunk
// c = k / (16 / element size)) sits at byte ((c * R/8) + g) * 128, so
// consecutive row groups are 128 B apart (SBO) and consecutive K chunks R*16 B
// apart (LBO). One MMA consumes 2 K chunks (K = 16 bf16 or 8 tf32); the k-th
// MMA's descriptor starts 2k chunks in.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "device_common.cuh"

namespace malib {
namespace tc {

// Byte offset of element (row, k) in the core-matrix layout of a tile with
// `rows` rows (multiple of 8) and elements of `es` bytes.
__host__ __device__ __forceinline__ uint32_t cm_offset(int row, int k, int rows, int es) {
    const int per_chunk = 16 / es;
    const int c = k / per_chunk, w = k % per_chunk;
    return (uint32_t)((c * (rows / 8) + (row >> 3)) * 128 + (row & 7) * 16 + w * es);
}

// Shared-memory matrix descriptor (tcgen05): start address, leading (K) and
// stride (row-group) byte offsets, all >> 4; bits 46-47 = 1; no swizzle.
__device__ __forceinline__ uint64_t smem_desc(uint32_t smem_addr, uint32_t lbo, uint32_t sbo) {
    uint64_t d = 0;
    d |= (uint64_t)((smem_addr >> 4) & 0x3FFFu);
    d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
    d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
    d |= (uint64_t)1 << 46;
    return d;
}

// Instruction descriptor, dense, D fp32, A and B K-major.
// ab_format: 1 = bf16 (kind::f16), 2 = tf32 (kind::tf32).
__host__ __device__ __forceinline__ uint32_t instr_desc(int M, int N, int ab_format) {
    uint32_t d = 0;
    d |= 1u << 4;                             // D format fp32
    d |= (uint32_t)ab_format << 7;            // A format
    d |= (uint32_t)ab_format << 10;           // B format
    d |= (uint32_t)(N >> 3) << 17;            // N / 8
    d |= (uint32_t)(M >> 4) << 24;            // M / 16
    return d;
}

// ---- tensor memory (one warp executes alloc / relinquish / dealloc) --------
__device__ __forceinline__ void tmem_alloc(uint32_t* smem_dst, uint32_t ncols) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(smem_dst)),
                 "r"(ncols)
                 : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
                 : "memory");
}

__device__ __forceinline__ void fence_before_sync() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void fence_after_sync() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// ---- MMA (issued by one thread) ---------------------------------------------
__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc,
                                         bool accumulate) {
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
        " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}" ::"r"(d_tmem),
        "l"(a), "l"(b), "r"(idesc), "r"((uint32_t)accumulate)
        : "memory");
}
__device__ __forceinline__ void mma_tf32(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc,
                                         bool accumulate) {
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
        " tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n}" ::"r"(d_tmem),
        "l"(a), "l"(b), "r"(idesc), "r"((uint32_t)accumulate)
        : "memory");
}
// Arrives on the mbarrier once every MMA issued so far by this thread is done.
__device__ __forceinline__ void mma_commit(uint64_t* bar) {
    asm volatile(
        "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
            smem_u32(bar))
        : "memory");
}

// ---- tensor memory -> registers: lanes of this warp's quarter, 32 columns ---
// A tcgen05.ld writes its destination registers asynchronously, until
// tcgen05.wait::ld. Every load here therefore sits in the same asm statement
// as its wait: the compiler never sees (and never reuses or spills) a
// destination register before its value has arrived.
// Two 32-column loads in flight together, then one wait.
__device__ __forceinline__ void tmem_ld32x2(uint32_t ta0, uint32_t ta1, uint32_t (&r0)[32],
                                            uint32_t (&r1)[32]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%64];\n"
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%32, %33, %34, %35, %36, %37, %38, %39, %40, %41, %42, %43, %44, %45, %46, %47, %48, %49, %50, %51, %52, %53, %54, %55, %56, %57, %58, %59, %60, %61, %62, %63}, [%65];\n"
        "tcgen05.wait::ld.sync.aligned;"
        : "=r"(r0[0]), "=r"(r0[1]), "=r"(r0[2]), "=r"(r0[3]),
          "=r"(r0[4]), "=r"(r0[5]), "=r"(r0[6]), "=r"(r0[7]),
          "=r"(r0[8]), "=r"(r0[9]), "=r"(r0[10]), "=r"(r0[11]),
          "=r"(r0[12]), "=r"(r0[13]), "=r"(r0[14]), "=r"(r0[15]),
          "=r"(r0[16]), "=r"(r0[17]), "=r"(r0[18]), "=r"(r0[19]),
          "=r"(r0[20]), "=r"(r0[21]), "=r"(r0[22]), "=r"(r0[23]),
          "=r"(r0[24]), "=r"(r0[25]), "=r"(r0[26]), "=r"(r0[27]),
          "=r"(r0[28]), "=r"(r0[29]), "=r"(r0[30]), "=r"(r0[31]),
          "=r"(r1[0]), "=r"(r1[1]), "=r"(r1[2]), "=r"(r1[3]),
          "=r"(r1[4]), "=r"(r1[5]), "=r"(r1[6]), "=r"(r1[7]),
          "=r"(r1[8]), "=r"(r1[9]), "=r"(r1[10]), "=r"(r1[11]),
          "=r"(r1[12]), "=r"(r1[13]), "=r"(r1[14]), "=r"(r1[15]),
          "=r"(r1[16]), "=r"(r1[17]), "=r"(r1[18]), "=r"(r1[19]),
          "=r"(r1[20]), "=r"(r1[21]), "=r"(r1[22]), "=r"(r1[23]),
          "=r"(r1[24]), "=r"(r1[25]), "=r"(r1[26]), "=r"(r1[27]),
          "=r"(r1[28]), "=r"(r1[29]), "=r"(r1[30]), "=r"(r1[31])
        : "r"(ta0), "r"(ta1)
        : "memory");
}

// One 32-column load as floats, completed in the same asm statement.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, "
        "%11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, "
        "%28, %29, %30, %31}, [%32];\n"
        "tcgen05.wait::ld.sync.aligned;"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
          "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]),
          "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
          "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]),
          "=r"(r[31])
        : "r"(taddr)
        : "memory");
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// One 32-column load (raw words), completed in the same asm statement.
__device__ __forceinline__ void tmem_ld32x1(uint32_t taddr, uint32_t (&r)[32]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, "
        "%11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, "
        "%28, %29, %30, %31}, [%32];\n"
        "tcgen05.wait::ld.sync.aligned;"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
          "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]),
          "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
          "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]),
          "=r"(r[31])
        : "r"(taddr)
        : "memory");
}

// One 16-column load as floats, completed in the same asm statement.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float (&v)[16]) {
    uint32_t r[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, "
        "%11, %12, %13, %14, %15}, [%16];\n"
        "tcgen05.wait::ld.sync.aligned;"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
          "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr)
        : "memory");
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// 16 lanes x 32 columns (shape 16x256b, four repeats), completed in the same
// asm statement. Thread T holds, for j = 0..3 (columns c = 8 j + 2 (T % 4)):
// r[4j] = (lane T/4, c), r[4j+1] = (lane T/4, c+1), r[4j+2] = (lane T/4 + 8, c),
// r[4j+3] = (lane T/4 + 8, c+1) - the layout of an mma.sync m16n8 accumulator,
// so that pairs of adjacent columns form an m16n8k16 A fragment.
__device__ __forceinline__ void tmem_ld16x256b_x4(uint32_t taddr, uint32_t (&r)[16]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.16x256b.x4.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, "
        "%11, %12, %13, %14, %15}, [%16];\n"
        "tcgen05.wait::ld.sync.aligned;"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
          "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr)
        : "memory");
}

// registers -> tensor memory: lanes of this warp's quarter, 16 columns. The
// caller issues tmem_wait_st() before the data may be read by an MMA.
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&r)[16]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, "
        "%11, %12, %13, %14, %15, %16};" ::"r"(taddr),
        "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
        "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]),
        "r"(r[15])
        : "memory");
}
__device__ __forceinline__ void tmem_wait_st() {
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

// bf16x2 of relu(x0) (low half) and relu(x1) (high half): rounding to
// nearest-even, negative results clamped to zero.
__device__ __forceinline__ uint32_t relu_bf16x2(float x0, float x1) {
    uint32_t r;
    asm("cvt.rn.relu.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(x1), "f"(x0));
    return r;
}

// TMEM address of (lane, column) given the allocation base.
__device__ __forceinline__ uint32_t tmem_addr(uint32_t base, int lane, int col) {
    return base + ((uint32_t)lane << 16) + (uint32_t)col;
}

// bf16 round-to-nearest-even of two floats packed low/high.
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
    uint32_t r;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
    return r;
}

// bf16x2 of relu(x0 + b0) (low half) and relu(x1 + b1) (high half): one packed
// fp32 add (each lane rounded to nearest, as a scalar add) and one conversion
// that rounds to nearest-even and clamps negative results to zero. Rounding is
// monotonic and keeps zero, so this equals rounding relu(x + b), up to the sign
// of a zero result.
__device__ __forceinline__ uint32_t bias_relu_bf16x2(float x0, float x1, float b0, float b1) {
    uint32_t r;
    asm("{\n .reg .b64 x, b, s;\n .reg .f32 lo, hi;\n"
        " mov.b64 x, {%1, %2};\n mov.b64 b, {%3, %4};\n"
        " add.rn.f32x2 s, x, b;\n"
        " mov.b64 {lo, hi}, s;\n"
        " cvt.rn.relu.bf16x2.f32 %0, hi, lo;\n}"
        : "=r"(r)
        : "f"(x0), "f"(x1), "f"(b0), "f"(b1));
    return r;
}

// setmaxnreg to R registers per thread in a kernel launched with kLaunch per
// thread: inc above the launch's count, dec below it, nothing at it (an inc to
// fewer registers, or a dec to more, is an illegal instruction). All threads
// of the warpgroup call it.
template <int R, int kLaunch>
__device__ __forceinline__ void set_max_regs() {
    static_assert(R % 8 == 0 && R >= 24 && R <= 256, "setmaxnreg's range");
    if constexpr (R > kLaunch) asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(R) : "memory");
    else if constexpr (R < kLaunch) asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(R) : "memory");
}

}  // namespace tc
}  // namespace malib
