// Population conversion on the device (Sec. 3.1 policy pools: the population
// arena the kernels read). Each policy's plain parameters, row-major W[out][in]
// then b[out] per layer in fp32, are copied into a staging buffer and gathered
// here into the policy's kernel image in the arena:
//   kind 0, table:  6 P(bet) values, 2 zeros;
//   kind 1, fp32:   W1T [in][h1] | b1 | W2T [h1][h2] | b2 | W3 [a][h2] | b3 | pad to 4
//                   (weights optionally rounded to bf16, biases kept fp32);
//   kind 2, bf16 tensor-core image: W1 [256][K1], W2 [256][256], W3 [16][256] as
//                   bf16 in the core-matrix K-major layout (8 rows x 16 bytes per
//                   core matrix, row groups 128 B apart, K chunks rows x 16 B
//                   apart), then fp32 b1 [256], b2 [256], b3 [16]; with the fold
//                   flag, input 15 (constant 1) is dropped and its bf16 weight
//                   added to b1.
// Every destination word is computed by one thread from its source values, so
// the image is the same whatever the launch shape. bf16 rounding is to
// nearest even on the bit pattern; infinities and NaNs keep their high half.
#include "internal.h"

namespace malib {

namespace {

__device__ __forceinline__ uint32_t bf16_bits(float x) {
    uint32_t b = __float_as_uint(x);
    if ((b & 0x7F800000u) != 0x7F800000u) b += 0x7FFFu + ((b >> 16) & 1u);
    return b >> 16;
}

__device__ __forceinline__ float bf16_value(float x) { return __uint_as_float(bf16_bits(x) << 16); }

// fp32 layout: the destination float i of a policy with dims d.
__device__ float f32_word(const float* p, const int* d, bool round, int64_t i) {
    const int64_t in = d[0], h1 = d[1], h2 = d[2], a = d[3];
    const float* W1 = p;
    const float* b1 = W1 + h1 * in;
    const float* W2 = b1 + h1;
    const float* b2 = W2 + h2 * h1;
    const float* W3 = b2 + h2;
    const float* b3 = W3 + a * h2;
    float v;
    bool weight = true;
    if (i < in * h1) {
        v = W1[(i % h1) * in + i / h1];
    } else if ((i -= in * h1) < h1) {
        v = b1[i];
        weight = false;
    } else if ((i -= h1) < h1 * h2) {
        v = W2[(i % h2) * h1 + i / h2];
    } else if ((i -= h1 * h2) < h2) {
        v = b2[i];
        weight = false;
    } else if ((i -= h2) < a * h2) {
        v = W3[i];
    } else if ((i -= a * h2) < a) {
        v = b3[i];
        weight = false;
    } else {
        return 0.f;
    }
    return round && weight ? bf16_value(v) : v;
}

// Tensor-core image: the destination 32-bit word i (two bf16 values of one
// core-matrix row, or one fp32 bias).
__device__ uint32_t tc_word(const float* p, const int* d, bool fold, int64_t i) {
    const int in = d[0], a = d[3];
    const int in_img = fold ? in - 1 : in;
    const int k1 = (in_img + 15) / 16 * 16;
    const float* W1 = p;
    const float* b1 = W1 + 256 * in;
    const float* W2 = b1 + 256;
    const float* b2 = W2 + 256 * 256;
    const float* W3 = b2 + 256;
    const float* b3 = W3 + a * 256;
    const int64_t n1 = 256 * k1 / 2, n2 = 256 * 256 / 2, n3 = 16 * 256 / 2;
    int region, rows;
    if (i < n1) {
        region = 1; rows = 256;
    } else if ((i -= n1) < n2) {
        region = 2; rows = 256;
    } else if ((i -= n2) < n3) {
        region = 3; rows = 16;
    } else {
        const int64_t j = i - n3;
        float v;
        if (j < 256) v = fold ? __fadd_rn(b1[j], bf16_value(W1[j * in + kLeducConstFeature])) : b1[j];
        else if (j < 512) v = b2[j - 256];
        else v = j - 512 < a ? b3[j - 512] : 0.f;
        return __float_as_uint(v);
    }
    // byte offset o inside the region -> (row, k) of its low half
    const int64_t o = 4 * i;
    const int64_t cm = o / 128;
    const int row = (int)((cm % (rows / 8)) * 8 + (o % 128) / 16);
    const int k = (int)((cm / (rows / 8)) * 8 + (o % 16) / 2);
    uint32_t h[2];
#pragma unroll
    for (int t = 0; t < 2; ++t) {
        const int kk = k + t;
        float v = 0.f;
        bool has = true;
        if (region == 1) {
            has = kk < in_img;
            if (has) v = W1[row * in + (fold && kk >= kLeducConstFeature ? kk + 1 : kk)];
        } else if (region == 2) {
            v = W2[row * 256 + kk];
        } else {
            has = row < a;
            if (has) v = W3[row * 256 + kk];
        }
        h[t] = has ? bf16_bits(v) : 0u;
    }
    return h[0] | (h[1] << 16);
}

__global__ void pop_convert_kernel(const ConvJob* __restrict__ jobs, const float* __restrict__ stage,
                                   float* __restrict__ arena) {
    const ConvJob j = jobs[blockIdx.y];
    const float* src = stage + j.src;
    uint32_t* dst = reinterpret_cast<uint32_t*>(arena + j.dst);
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < j.size;
         i += (int64_t)gridDim.x * blockDim.x) {
        uint32_t w;
        if (j.kind == kConvTable) w = __float_as_uint(i < 6 ? src[i] : 0.f);
        else if (j.kind == kConvF32) w = __float_as_uint(f32_word(src, j.dims, (j.flags & kConvRound) != 0, i));
        else w = tc_word(src, j.dims, (j.flags & kConvFold) != 0, i);
        dst[i] = w;
    }
}

}  // namespace

cudaError_t launch_pop_convert(const ConvJob* jobs, int n_jobs, int64_t max_size, const float* stage,
                               float* arena, cudaStream_t s) {
    if (n_jobs <= 0) return cudaSuccess;
    if (n_jobs > 65535) return cudaErrorInvalidValue;
    const int64_t bx = (max_size + 255) / 256;
    const unsigned gx = (unsigned)(bx < 64 ? (bx < 1 ? 1 : bx) : 64);
    pop_convert_kernel<<<dim3(gx, (unsigned)n_jobs), 256, 0, s>>>(jobs, stage, arena);
    return cudaGetLastError();
}

}  // namespace malib
