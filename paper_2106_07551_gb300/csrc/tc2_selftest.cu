// The pipelined tensor-core policy forward (mlp_tc2.cuh) on its own: rows of
// observations through one policy of a loaded bf16 population, logits out.
// It checks the engine against an fp64 forward with bf16 rounding (the parity
// tests) and measures its rate on resident inputs (the engine's roofline).
//
// One persistent CTA per SM, tiles of 128 rows dealt round robin; `reps`
// repeats the row set (the same logits are written again), so a small input
// gives a long, compute-only run. The engine's warps come first (two
// epilogue teams of kTW warps, two MMA warps); the last four warps convert
// rows to a bf16 observation tile (one row per thread) and, two tiles behind,
// add each row's partial logits and b3 and store them.
#include "device_common.cuh"
#include "internal.h"
#include "malib.h"
#include "mlp_tc2.cuh"

namespace malib {

namespace {

constexpr int kTW = 8;                       // epilogue warps per slot
constexpr int kIoWarp = 4 * kTW / 2 + 2;     // after both teams and the two MMA warps
constexpr int kThreads = (kIoWarp + 4) * 32;
constexpr uint32_t kLag = 2;                 // results of tile i are taken after producing tile i + 2

template <int K1, int A>
struct ProbeLayout {
    using E = Eng2<K1, A, 3, kTW>;
    static constexpr uint32_t kX = (E::kImage + 1023u) / 1024u * 1024u;
    static constexpr uint32_t kP = kX + E::kNX * E::kXBytes;
    static constexpr uint32_t kSmem = kP + 2 * E::kPBytes;
    static_assert(kSmem <= 227u * 1024u, "fits one CTA's shared memory");
};

template <int K1, int A, bool kFold>
__global__ void __launch_bounds__(kThreads, 1)
    mlp_tc2_probe_kernel(const float* __restrict__ arena, const int64_t* __restrict__ pol_offset,
                         int32_t pid, const float* __restrict__ x,
                         int in, int64_t n_rows, int32_t reps, float* __restrict__ out, int* err) {
    using E = Eng2<K1, A, 3, kTW>;
    using L = ProbeLayout<K1, A>;
    extern __shared__ __align__(1024) uint8_t smem[];
    __shared__ typename E::Bars bars;
    __shared__ uint32_t tmem_base;
    const int tid = threadIdx.x, warp = tid >> 5;

    if (tid == 0) {
        bars.init();
        E::stage(smem, reinterpret_cast<const uint8_t*>(arena + pol_offset[pid]), bars);
    }
    if (warp == 0) {
        tc::tmem_alloc(&tmem_base, E::kTmemCols);
        tc::tmem_relinquish();
    }
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    const uint32_t tbase = tmem_base;
    const int64_t row_tiles = (n_rows + 127) / 128;
    const int64_t tiles = row_tiles * reps;
    const uint32_t n = (uint32_t)((tiles - blockIdx.x + gridDim.x - 1) / gridDim.x);

    if (warp < kTW) {
        typename E::template Epilogue<0> ep;
        ep.p_base_off = L::kP;
        E::wait(bars, &bars.stage, 0u, err);
        ep.init(smem);
        ep.run(smem, tbase, bars, n, err);
    } else if (warp < E::kEpiWarps) {
        typename E::template Epilogue<1> ep;
        ep.p_base_off = L::kP;
        E::wait(bars, &bars.stage, 0u, err);
        ep.init(smem);
        ep.run(smem, tbase, bars, n, err);
    } else if (warp == E::kIssuerWarp) {
        if ((tid & 31) == 0) {
            typename E::template Issuer<0> is;
            E::wait(bars, &bars.stage, 0u, err);
            is.run(smem, smem_u32(smem + L::kX), tbase, bars, n, err);
            is.finish(bars, err);
        }
    } else if (warp == E::kIssuerWarp + 1) {
        if ((tid & 31) == 0) {
            typename E::template Issuer<1> is;
            E::wait(bars, &bars.stage, 0u, err);
            is.run(smem, smem_u32(smem + L::kX), tbase, bars, n, err);
            is.finish(bars, err);
        }
    } else {
        const int r = tid - kIoWarp * 32;                 // row of the tile
        E::wait(bars, &bars.stage, 0u, err);
        const float* b3 = reinterpret_cast<const float*>(smem + E::kB3);
        for (uint32_t i = 0; i < n + kLag; ++i) {
            if (i < n) {
                const int64_t tile = (int64_t)blockIdx.x + (int64_t)i * gridDim.x;
                const int64_t row = (tile % row_tiles) * 128 + r;
                const int buf = (int)(i % E::kNX);
                if (i >= (uint32_t)E::kNX) E::wait(bars, &bars.x_free[buf], ((i / E::kNX) - 1) & 1u, err);
                uint8_t* xt = smem + L::kX + buf * E::kXBytes;
#pragma unroll
                for (int c = 0; c < K1 / 8; ++c) {
                    uint32_t w[4];
#pragma unroll
                    for (int h = 0; h < 4; ++h) {
                        float v[2];
#pragma unroll
                        for (int e = 0; e < 2; ++e) {
                            const int k = 8 * c + 2 * h + e;                  // image input slot
                            const int f = kFold && k >= kLeducConstFeature ? k + 1 : k;   // feature
                            v[e] = (row < n_rows && f < in) ? x[row * in + f] : 0.f;
                        }
                        w[h] = tc::pack_bf16(v[0], v[1]);
                    }
                    *reinterpret_cast<uint4*>(xt + E::x_offset(r, 8 * c)) = make_uint4(w[0], w[1], w[2], w[3]);
                }
                fence_proxy_async_smem();
                asm volatile("bar.sync 2, 128;" ::: "memory");
                if (r == 0) mbar_arrive_release(&bars.x_full[buf]);
            }
            if (i >= kLag) {
                const uint32_t c = i - kLag;
                const int64_t tile = (int64_t)blockIdx.x + (int64_t)c * gridDim.x;
                const int64_t row = (tile % row_tiles) * 128 + r;
                const int sl = (int)(c & 1u);
                E::wait(bars, &bars.p_full[sl], (c >> 1) & 1u, err);
                const float* p = reinterpret_cast<const float*>(smem + L::kP + sl * E::kPBytes);
                if (row < n_rows) {
#pragma unroll
                    for (int a = 0; a < A; ++a) {
                        float v = p[r * A + a];
                        if (E::kSplit == 2) v = __fadd_rn(v, p[(128 + r) * A + a]);
                        out[row * A + a] = __fadd_rn(v, b3[a]);
                    }
                }
                asm volatile("bar.sync 2, 128;" ::: "memory");
                if (r == 0) mbar_arrive_release(&bars.p_free[sl]);
            }
        }
    }
    tc::fence_before_sync();
    __syncthreads();
    if (warp == 0) tc::tmem_dealloc(tbase, E::kTmemCols);
}

template <int K1, int A, bool kFold>
cudaError_t launch_probe(const float* arena, const int64_t* off, int32_t pid, const float* x, int in,
                         int64_t n_rows,
                         int32_t reps, float* out, int* err, int n_sm, cudaStream_t s) {
    using L = ProbeLayout<K1, A>;
    auto k = mlp_tc2_probe_kernel<K1, A, kFold>;
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)L::kSmem);
    if (e != cudaSuccess) return e;
    const int64_t tiles = (n_rows + 127) / 128 * reps;
    const unsigned grid = (unsigned)(tiles < n_sm ? tiles : n_sm);
    k<<<grid, kThreads, L::kSmem, s>>>(arena, off, pid, x, in, n_rows, reps, out, err);
    return cudaGetLastError();
}

}  // namespace

}  // namespace malib

using namespace malib;

extern "C" int malib_selftest_mlp_tc(malib_ctx* ctx, int32_t policy_id, const float* x, int64_t n_rows,
                                     int32_t reps, float* logits_out) {
    CtxView v;
    if (!ctx_view(ctx, &v)) return MALIB_EINVAL;
    if (!v.has_pop || !v.tc_layout) return ctx_fail(ctx, MALIB_ESTATE, "no bf16 tensor-core population loaded");
    if (policy_id < 0 || policy_id >= v.n_pol) return ctx_fail(ctx, MALIB_EINVAL, "policy id out of range");
    if (n_rows < 0 || reps < 1) return ctx_fail(ctx, MALIB_EINVAL, "n_rows < 0 or reps < 1");
    if (n_rows == 0) return MALIB_OK;
    if (ptr_where(x, v.device) != kPtrHere || ptr_where(logits_out, v.device) != kPtrHere)
        return ctx_fail(ctx, MALIB_EINVAL, "x and logits_out must be device memory of the context's device");
    if (n_rows > ((int64_t)1 << 31) / 64) return ctx_fail(ctx, MALIB_EINVAL, "n_rows too large");
    const bool leduc = v.env_kind == MALIB_ENV_LEDUC && v.dims[0] == 17 && v.dims[3] == 3;
    const bool spread = v.dims[0] == 34 && v.dims[3] == 5;
    if (!leduc && !spread)
        return ctx_fail(ctx, MALIB_EUNSUPPORTED, "engine probe built for 17-256-256-3 (Leduc) and 34-256-256-5");
    int prev = -1;
    if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
    if (cudaSetDevice(v.device) != cudaSuccess) return ctx_fail(ctx, MALIB_ECUDA, "cannot select the device");
    const cudaError_t e =
        leduc ? launch_probe<16, 3, true>(v.arena, v.pol_offset, policy_id, x, 17, n_rows, reps, logits_out, v.err, v.n_sm, v.stream)
              : launch_probe<48, 5, false>(v.arena, v.pol_offset, policy_id, x, 34, n_rows, reps, logits_out, v.err, v.n_sm, v.stream);
    if (prev >= 0) cudaSetDevice(prev);
    if (e != cudaSuccess) return ctx_fail(ctx, MALIB_ECUDA, cudaGetErrorString(e));
    ctx_count_launches(ctx, 1);
    return MALIB_OK;
}
