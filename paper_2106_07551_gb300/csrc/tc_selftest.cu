// Self-test of the tensor-core building blocks: one CTA computes
// D[128][N] = A[128][K] . B[N][K]^T with tcgen05 MMAs from shared memory (bf16 or
// tf32 operands, fp32 accumulator in tensor memory), exactly the operand
// layout, descriptors and completion path the MLP kernels use.
#include "device_common.cuh"
#include "internal.h"
#include "malib.h"
#include "tc_common.cuh"

namespace malib {

namespace {

template <bool TF32>
__global__ void __launch_bounds__(128, 1) mma_selftest_kernel(const void* A, const void* B,
                                                              float* D, int N, int K,
                                                              uint32_t ncols, int* err) {
    constexpr int es = TF32 ? 4 : 2;
    extern __shared__ __align__(1024) uint8_t smem[];
    __shared__ __align__(8) uint64_t bar;
    __shared__ uint32_t tmem_base;
    uint8_t* sA = smem;
    uint8_t* sB = smem + 128 * K * es;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

    for (int k = 0; k < K; ++k) {
        const uint8_t* src = (const uint8_t*)A + ((size_t)tid * K + k) * es;
        uint8_t* dst = sA + tc::cm_offset(tid, k, 128, es);
        for (int b = 0; b < es; ++b) dst[b] = src[b];
    }
    for (int n = tid; n < N; n += 128)
        for (int k = 0; k < K; ++k) {
            const uint8_t* src = (const uint8_t*)B + ((size_t)n * K + k) * es;
            uint8_t* dst = sB + tc::cm_offset(n, k, N, es);
            for (int b = 0; b < es; ++b) dst[b] = src[b];
        }
    if (tid == 0) mbar_init(&bar, 1);
    fence_proxy_async_smem();
    __syncthreads();
    if (warp == 0) {
        tc::tmem_alloc(&tmem_base, ncols);
        tc::tmem_relinquish();
    }
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    const uint32_t tbase = tmem_base;

    if (tid == 0) {
        const uint32_t idesc = tc::instr_desc(128, N, TF32 ? 2 : 1);
        const uint32_t lbo_a = (128 / 8) * 128, lbo_b = (uint32_t)(N / 8) * 128;
        const int steps = K / (TF32 ? 8 : 16);
        for (int s = 0; s < steps; ++s) {
            const uint64_t da = tc::smem_desc(smem_u32(sA) + 2u * s * lbo_a, lbo_a, 128);
            const uint64_t db = tc::smem_desc(smem_u32(sB) + 2u * s * lbo_b, lbo_b, 128);
            if (TF32) tc::mma_tf32(tbase, da, db, idesc, s > 0);
            else tc::mma_bf16(tbase, da, db, idesc, s > 0);
        }
        tc::mma_commit(&bar);
    }
    const bool ok = mbar_wait_bounded(&bar, 0, kWaitLimitNs);
    tc::fence_after_sync();
    if (!ok) {
        if (tid == 0) atomicOr(err, ERRBIT_TIMEOUT);
    } else {
        for (int c0 = 0; c0 < N; c0 += 32) {
            float v[32];
            tc::tmem_ld32(tc::tmem_addr(tbase, 32 * warp, c0), v);
            float* out = D + (size_t)(32 * warp + lane) * N + c0;
#pragma unroll
            for (int i = 0; i < 32; ++i)
                if (c0 + i < N) out[i] = v[i];   // N may be 16: columns past N are not D's
        }
    }
    tc::fence_before_sync();
    __syncthreads();
    if (warp == 0) tc::tmem_dealloc(tbase, ncols);
}

bool device_ptr(const void* p) {
    cudaPointerAttributes at;
    if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    return at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged;
}

}  // namespace

}  // namespace malib

using namespace malib;

extern "C" int malib_selftest_mma(malib_ctx* ctx, int32_t dtype, const void* A, const void* B,
                                  float* D, int32_t N, int32_t K) {
    CtxView v;
    if (!ctx_view(ctx, &v)) return MALIB_EINVAL;
    const bool tf32 = dtype == MALIB_F32;
    if (dtype != MALIB_F32 && dtype != MALIB_BF16)
        return ctx_fail(ctx, MALIB_EINVAL, "dtype must be MALIB_BF16 or MALIB_F32 (tf32 MMA)");
    const int es = tf32 ? 4 : 2;
    if (N < 16 || N > 256 || N % 16 != 0)
        return ctx_fail(ctx, MALIB_EINVAL, "N must be a multiple of 16 in [16, 256]");
    if (K < 1 || K % (tf32 ? 8 : 16) != 0)
        return ctx_fail(ctx, MALIB_EINVAL, "K must be a multiple of the MMA K (16 bf16, 8 tf32)");
    const size_t bytes = (size_t)(128 + N) * K * es;
    if (bytes > 200 * 1024) return ctx_fail(ctx, MALIB_EINVAL, "operands exceed 200 KB of shared memory");
    if (!A || !B || !D || !device_ptr(A) || !device_ptr(B) || !device_ptr(D))
        return ctx_fail(ctx, MALIB_EINVAL, "A, B and D must be device buffers");
    uint32_t ncols = 32;
    while (ncols < (uint32_t)N) ncols <<= 1;
    int prev = -1;
    if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
    cudaSetDevice(v.device);
    cudaError_t e;
    if (tf32) {
        e = cudaFuncSetAttribute(mma_selftest_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)bytes);
        if (e == cudaSuccess) {
            mma_selftest_kernel<true><<<1, 128, bytes, v.stream>>>(A, B, D, N, K, ncols, v.err);
            e = cudaGetLastError();
        }
    } else {
        e = cudaFuncSetAttribute(mma_selftest_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)bytes);
        if (e == cudaSuccess) {
            mma_selftest_kernel<false><<<1, 128, bytes, v.stream>>>(A, B, D, N, K, ncols, v.err);
            e = cudaGetLastError();
        }
    }
    if (prev >= 0) cudaSetDevice(prev);
    if (e != cudaSuccess) return ctx_fail(ctx, MALIB_ECUDA, cudaGetErrorString(e));
    ctx_count_launches(ctx, 1);
    return MALIB_OK;
}
