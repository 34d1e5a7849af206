// Small kernels around the main ones: zeroing the payoff sums, turning them
// into payoff-table entries, and self-test entry points that expose the
// sampling primitives every kernel uses.
#include "device_common.cuh"
#include "internal.h"

namespace malib {

namespace {

__global__ void zero_u64_kernel(unsigned long long* p, int64_t n) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x)
        p[i] = 0ull;
}

// Entry of the payoff table (Sec. 3.2) from the integer sums of n hands:
// mean, standard error of the mean (sample variance with n - 1; 0 if n < 2),
// sum and sum of squares.
__global__ void finalize_kernel(const unsigned long long* acc, int32_t n_pairs, int64_t n,
                                double* out) {
    const int p = blockIdx.x * blockDim.x + threadIdx.x;
    if (p >= n_pairs) return;
    finalize_pair((long long)acc[2 * p], (long long)acc[2 * p + 1], n, out + 4 * p);
}

__global__ void philox_kernel(const uint32_t* ctr, uint64_t seed, uint32_t* out, int64_t n) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x) {
        const uint4 c = reinterpret_cast<const uint4*>(ctr)[i];
        const U4 r = philox10(c.x, c.y, c.z, c.w, (uint32_t)seed, (uint32_t)(seed >> 32));
        reinterpret_cast<uint4*>(out)[i] = make_uint4(r.x, r.y, r.z, r.w);
    }
}

// Philox throughput probe: thread t XOR-folds the four words of the calls
// i = 0..calls-1 at counter (t lo, t hi, i, 0) into out[t]. One 4-byte store
// per thread, so the time is the generator's arithmetic.
__global__ void __launch_bounds__(256) philox_digest_kernel(uint64_t seed, int64_t n, int calls,
                                                            uint32_t* out) {
    const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (t >= n) return;
    const uint32_t k0 = (uint32_t)seed, k1 = (uint32_t)(seed >> 32);
    uint32_t acc = 0u;
#pragma unroll 4
    for (int i = 0; i < calls; ++i) {
        const U4 r = philox10((uint32_t)t, (uint32_t)(t >> 32), (uint32_t)i, 0u, k0, k1);
        acc ^= r.x ^ r.y ^ r.z ^ r.w;
    }
    out[t] = acc;
}

// Bounded-wait self-test: one thread waits at most limit_ns for the first
// phase of an mbarrier of count 1 that it arrives on itself (arrive) or that
// nothing arrives on; an expired wait sets ERRBIT_TIMEOUT and the kernel ends.
__global__ void wait_selftest_kernel(bool arrive, uint64_t limit_ns, int* err) {
    __shared__ __align__(8) uint64_t bar;
    if (threadIdx.x != 0) return;
    mbar_init(&bar, 1);
    if (arrive) mbar_arrive_release(&bar);
    if (!mbar_wait_bounded(&bar, 0, limit_ns)) atomicOr(err, ERRBIT_TIMEOUT);
}

__global__ void det_expf_kernel(const float* x, float* y, int64_t n) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x)
        y[i] = det_expf(x[i]);
}

template <int A>
__global__ void sample_kernel(const float* logits, const uint8_t* legal, const float* u,
                              int32_t* out, int64_t n) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x) {
        float lg[A];
        unsigned bits = 0;
#pragma unroll
        for (int a = 0; a < A; ++a) {
            lg[a] = logits[i * A + a];
            bits |= legal[i * A + a] ? (1u << a) : 0u;
        }
        out[i] = sample_masked<A>(lg, bits, u[i]);
    }
}

unsigned grid_for(int64_t n, int threads) {
    int64_t b = (n + threads - 1) / threads;
    if (b > 4096) b = 4096;
    return (unsigned)(b < 1 ? 1 : b);
}

}  // namespace

cudaError_t launch_zero_u64(unsigned long long* p, int64_t n, cudaStream_t s) {
    if (n <= 0) return cudaSuccess;
    zero_u64_kernel<<<grid_for(n, 256), 256, 0, s>>>(p, n);
    return cudaGetLastError();
}

cudaError_t launch_finalize(const unsigned long long* acc, int32_t n_pairs, int64_t n_episodes,
                            double* out, cudaStream_t s) {
    if (n_pairs <= 0) return cudaSuccess;
    finalize_kernel<<<(n_pairs + 127) / 128, 128, 0, s>>>(acc, n_pairs, n_episodes, out);
    return cudaGetLastError();
}

cudaError_t launch_selftest_philox(const uint32_t* ctr, uint64_t seed, uint32_t* out, int64_t n,
                                   cudaStream_t s) {
    if (n <= 0) return cudaSuccess;
    philox_kernel<<<grid_for(n, 256), 256, 0, s>>>(ctr, seed, out, n);
    return cudaGetLastError();
}

cudaError_t launch_philox_digest(uint64_t seed, int64_t n, int calls, uint32_t* out,
                                 cudaStream_t s) {
    if (n <= 0) return cudaSuccess;
    const int64_t blocks = (n + 255) / 256;
    if (blocks > 0x7FFFFFFF) return cudaErrorInvalidValue;
    philox_digest_kernel<<<(unsigned)blocks, 256, 0, s>>>(seed, n, calls, out);
    return cudaGetLastError();
}

cudaError_t launch_selftest_wait(bool arrive, uint64_t limit_ns, int* err, cudaStream_t s) {
    wait_selftest_kernel<<<1, 32, 0, s>>>(arrive, limit_ns, err);
    return cudaGetLastError();
}

cudaError_t launch_selftest_det_expf(const float* x, float* y, int64_t n, cudaStream_t s) {
    if (n <= 0) return cudaSuccess;
    det_expf_kernel<<<grid_for(n, 256), 256, 0, s>>>(x, y, n);
    return cudaGetLastError();
}

cudaError_t launch_selftest_sample(const float* logits, const uint8_t* legal, const float* u,
                                   int A, int32_t* out, int64_t n, cudaStream_t s) {
    if (n <= 0) return cudaSuccess;
    const unsigned g = grid_for(n, 256);
    switch (A) {
        case 2: sample_kernel<2><<<g, 256, 0, s>>>(logits, legal, u, out, n); break;
        case 3: sample_kernel<3><<<g, 256, 0, s>>>(logits, legal, u, out, n); break;
        case 4: sample_kernel<4><<<g, 256, 0, s>>>(logits, legal, u, out, n); break;
        case 5: sample_kernel<5><<<g, 256, 0, s>>>(logits, legal, u, out, n); break;
        case 6: sample_kernel<6><<<g, 256, 0, s>>>(logits, legal, u, out, n); break;
        case 7: sample_kernel<7><<<g, 256, 0, s>>>(logits, legal, u, out, n); break;
        case 8: sample_kernel<8><<<g, 256, 0, s>>>(logits, legal, u, out, n); break;
        default: return cudaErrorInvalidValue;
    }
    return cudaGetLastError();
}

}  // namespace malib
