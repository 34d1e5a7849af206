// Meta-game solvers on the payoff table (Sec. 4.2: the PSRO loop on Leduc uses
// fictitious play as its meta-solver and names an exact LP solver; App. C.2:
// payoffs aggregated under the equilibrium). A[i][j] is seat 0's payoff when
// row policy i meets column policy j; the games are zero-sum.
//
// One CTA solves one game (batched over a grid of games). Everything a game
// needs stays on chip: the payoff matrix (or the LP tableau) in shared memory
// when it fits, cumulative payoffs in registers, and each iteration's argmax /
// argmin in warp shuffles plus one cross-warp step.
#include <cstdint>

#include "internal.h"
#include "malib.h"

namespace malib {

namespace {

constexpr int kFpThreads = 256;
constexpr int kFpPer = 4;                       // rows (columns) per thread: m, n <= 1024
constexpr int kFpMaxDim = kFpThreads * kFpPer;
constexpr int kSmemLimit = 200 * 1024;          // bytes of payoff / tableau kept on chip

struct ArgBest {
    double v;
    int i;
};

// Better of two candidates: larger (sign = +1) or smaller (sign = -1) value,
// the lower index on equal values.
__device__ __forceinline__ ArgBest better(ArgBest a, ArgBest b, double sign) {
    const double av = sign * a.v, bv = sign * b.v;
    if (b.i < 0) return a;
    if (a.i < 0) return b;
    if (bv > av || (bv == av && b.i < a.i)) return b;
    return a;
}

__device__ __forceinline__ ArgBest warp_best(ArgBest a, double sign) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        ArgBest b;
        b.v = __shfl_xor_sync(0xffffffffu, a.v, o);
        b.i = __shfl_xor_sync(0xffffffffu, a.i, o);
        a = better(a, b, sign);
    }
    return a;
}

// Simultaneous fictitious play: both play policy 0 first; then each plays the
// first best response to the other's plays so far. u_row[i] = sum over plays
// of A[i][j_s] and u_col[j] = sum of A[i_s][j] are fp64 sums in play order.
__global__ void __launch_bounds__(kFpThreads) fictitious_play_kernel(
    const double* __restrict__ P, int32_t n_games, int32_t m, int32_t n, int32_t stride,
    int64_t T, double* __restrict__ x_out, double* __restrict__ y_out,
    double* __restrict__ bounds_out, int32_t on_chip) {
    extern __shared__ double sA[];              // [m][ld] when on chip
    __shared__ ArgBest red[2][kFpThreads / 32];
    __shared__ int play[2];
    __shared__ long long cnt_row[kFpMaxDim], cnt_col[kFpMaxDim];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int ld = n | 1;                       // odd row stride: column reads hit distinct banks

    for (int g = blockIdx.x; g < n_games; g += gridDim.x) {
        const double* Pg = P + (int64_t)g * m * n * stride;
        if (on_chip) {
            for (int k = tid; k < m * n; k += kFpThreads) {
                const int i = k / n, j = k - i * n;
                sA[i * ld + j] = Pg[(int64_t)k * stride];
            }
        }
        for (int k = tid; k < kFpMaxDim; k += kFpThreads) { cnt_row[k] = 0; cnt_col[k] = 0; }
        if (tid == 0) { play[0] = 0; play[1] = 0; }
        __syncthreads();
        auto a_at = [&](int i, int j) -> double {
            return on_chip ? sA[i * ld + j] : __ldg(Pg + ((int64_t)i * n + j) * stride);
        };
        double ur[kFpPer], uc[kFpPer];
#pragma unroll
        for (int k = 0; k < kFpPer; ++k) { ur[k] = 0.0; uc[k] = 0.0; }
        ArgBest top{0.0, -1}, bot{0.0, -1};
        for (int64_t t = 0; t < T; ++t) {
            const int it = play[0], jt = play[1];
            if (tid == 0) { cnt_row[it] += 1; cnt_col[jt] += 1; }
            ArgBest br{0.0, -1}, bc{0.0, -1};
#pragma unroll
            for (int k = 0; k < kFpPer; ++k) {
                const int i = tid + k * kFpThreads;
                if (i < m) {
                    ur[k] += a_at(i, jt);
                    br = better(br, ArgBest{ur[k], i}, 1.0);
                }
                if (i < n) {
                    uc[k] += a_at(it, i);
                    bc = better(bc, ArgBest{uc[k], i}, -1.0);
                }
            }
            br = warp_best(br, 1.0);
            bc = warp_best(bc, -1.0);
            if (lane == 0) { red[0][warp] = br; red[1][warp] = bc; }
            __syncthreads();                    // also: every thread has read play[]
            if (warp == 0) {
                ArgBest r = lane < kFpThreads / 32 ? red[0][lane] : ArgBest{0.0, -1};
                ArgBest c = lane < kFpThreads / 32 ? red[1][lane] : ArgBest{0.0, -1};
                r = warp_best(r, 1.0);
                c = warp_best(c, -1.0);
                if (lane == 0) { play[0] = r.i; play[1] = c.i; top = r; bot = c; }
            }
            __syncthreads();
        }
        const double Td = (double)T;
        for (int i = tid; i < m; i += kFpThreads) x_out[(int64_t)g * m + i] = (double)cnt_row[i] / Td;
        for (int j = tid; j < n; j += kFpThreads) y_out[(int64_t)g * n + j] = (double)cnt_col[j] / Td;
        if (tid == 0) {
            bounds_out[2 * g] = bot.v / Td;     // min_j (x^T A)_j
            bounds_out[2 * g + 1] = top.v / Td; // max_i (A y)_i
        }
        __syncthreads();
    }
}

// Payoffs under a pair of mixtures: A y (per row), x^T A (per column), x^T A y.
__global__ void __launch_bounds__(256) aggregate_kernel(
    const double* __restrict__ P, int32_t n_games, int32_t m, int32_t n, int32_t stride,
    const double* __restrict__ x, const double* __restrict__ y, double* __restrict__ ay_out,
    double* __restrict__ xa_out, double* __restrict__ val_out) {
    __shared__ double red[8];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    for (int g = blockIdx.x; g < n_games; g += gridDim.x) {
        const double* Pg = P + (int64_t)g * m * n * stride;
        const double* xg = x + (int64_t)g * m;
        const double* yg = y + (int64_t)g * n;
        double part = 0.0;
        for (int i = tid; i < m; i += blockDim.x) {
            double s = 0.0;
            for (int j = 0; j < n; ++j) s = fma(Pg[((int64_t)i * n + j) * stride], yg[j], s);
            ay_out[(int64_t)g * m + i] = s;
            part = fma(xg[i], s, part);
        }
        for (int j = tid; j < n; j += blockDim.x) {
            double s = 0.0;
            for (int i = 0; i < m; ++i) s = fma(xg[i], Pg[((int64_t)i * n + j) * stride], s);
            xa_out[(int64_t)g * n + j] = s;
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) part += __shfl_xor_sync(0xffffffffu, part, o);
        if (lane == 0) red[warp] = part;
        __syncthreads();
        if (tid == 0) {
            double v = 0.0;
            for (int w = 0; w < (int)(blockDim.x >> 5); ++w) v += red[w];
            val_out[g] = v;
        }
        __syncthreads();
    }
}

// ---------------------------------------------------------------------------
// Exact equilibrium by the simplex method. With B = A - min(A) + 1 > 0, the
// column player's problem max sum(q) s.t. B q <= 1, q >= 0 has optimum
// 1 / v_B; y = q v_B, and the row player's x = p v_B from the duals p (the
// objective row under the slack columns). v_A = v_B + min(A) - 1.
// Tableau rows 0..m-1: [B | I | 1]; row m: [-1 ... -1 | 0 | 0]. Bland's rule
// (lowest entering index with a negative reduced cost; lowest basic index on
// ratio ties) guarantees termination; a pivot limit guards regardless.
// ---------------------------------------------------------------------------
constexpr int kLpThreads = 512;

__global__ void __launch_bounds__(kLpThreads) lp_nash_kernel(
    const double* __restrict__ P, int32_t n_games, int32_t m, int32_t n, int32_t stride,
    double* __restrict__ x_out, double* __restrict__ y_out, double* __restrict__ val_out,
    double* __restrict__ gscratch, int32_t on_chip, int* __restrict__ err) {
    extern __shared__ double smem_tab[];
    __shared__ double colq[1024 + 1];
    __shared__ int basis[1024];
    __shared__ ArgBest red[kLpThreads / 32];
    __shared__ int enter_s, leave_s;
    __shared__ double amin_s;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int W = n + m + 1;                     // tableau width; column W-1 is the right side
    const int H = m + 1;                         // rows; row m is the objective

    for (int g = blockIdx.x; g < n_games; g += gridDim.x) {
        double* Tb = on_chip ? smem_tab : gscratch + (int64_t)blockIdx.x * H * W;
        const double* Pg = P + (int64_t)g * m * n * stride;
        // min(A)
        ArgBest lo{0.0, -1};
        for (int k = tid; k < m * n; k += kLpThreads) lo = better(lo, ArgBest{Pg[(int64_t)k * stride], k}, -1.0);
        lo = warp_best(lo, -1.0);
        if (lane == 0) red[warp] = lo;
        __syncthreads();
        if (warp == 0) {
            ArgBest r = lane < kLpThreads / 32 ? red[lane] : ArgBest{0.0, -1};
            r = warp_best(r, -1.0);
            if (lane == 0) amin_s = r.v;
        }
        __syncthreads();
        const double shift = 1.0 - amin_s;
        for (int k = tid; k < H * W; k += kLpThreads) {
            const int r = k / W, c = k - r * W;
            double v;
            if (r < m) {
                if (c < n) v = Pg[((int64_t)r * n + c) * stride] + shift;
                else if (c < n + m) v = (c - n == r) ? 1.0 : 0.0;
                else v = 1.0;
            } else {
                v = c < n ? -1.0 : 0.0;
            }
            Tb[k] = v;
        }
        for (int r = tid; r < m; r += kLpThreads) basis[r] = n + r;
        __syncthreads();

        const int max_pivots = 50 * (m + n) + 1000;
        bool done = false;
        for (int piv = 0; piv < max_pivots; ++piv) {
            // entering column: lowest index with a negative reduced cost
            const double eps = 1e-12;
            int ent = 0x7fffffff;
            for (int c = tid; c < n + m; c += kLpThreads)
                if (Tb[(int64_t)m * W + c] < -eps) { ent = c; break; }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) ent = min(ent, __shfl_xor_sync(0xffffffffu, ent, o));
            if (lane == 0) red[warp].i = ent;
            __syncthreads();
            if (tid == 0) {
                int e = 0x7fffffff;
                for (int w = 0; w < kLpThreads / 32; ++w) e = min(e, red[w].i);
                enter_s = e;
            }
            __syncthreads();
            const int q = enter_s;
            if (q == 0x7fffffff) { done = true; break; }
            // ratio test over rows with a positive pivot-column entry; ties to
            // the lowest basic variable index
            ArgBest best{0.0, -1};
            int best_basis = 0x7fffffff;
            for (int r = tid; r < m; r += kLpThreads) {
                const double a = Tb[(int64_t)r * W + q];
                if (a > eps) {
                    const double ratio = Tb[(int64_t)r * W + W - 1] / a;
                    if (best.i < 0 || ratio < best.v || (ratio == best.v && basis[r] < best_basis)) {
                        best = ArgBest{ratio, r};
                        best_basis = basis[r];
                    }
                }
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) {
                const double ov = __shfl_xor_sync(0xffffffffu, best.v, o);
                const int oi = __shfl_xor_sync(0xffffffffu, best.i, o);
                const int ob = __shfl_xor_sync(0xffffffffu, best_basis, o);
                if (oi >= 0 && (best.i < 0 || ov < best.v || (ov == best.v && ob < best_basis))) {
                    best = ArgBest{ov, oi};
                    best_basis = ob;
                }
            }
            if (lane == 0) red[warp] = best;
            __syncthreads();
            if (tid == 0) {
                ArgBest b{0.0, -1};
                int bb = 0x7fffffff;
                for (int w = 0; w < kLpThreads / 32; ++w) {
                    const ArgBest o = red[w];
                    if (o.i < 0) continue;
                    const int ob = basis[o.i];
                    if (b.i < 0 || o.v < b.v || (o.v == b.v && ob < bb)) { b = o; bb = ob; }
                }
                leave_s = b.i;                   // -1: unbounded (cannot happen with B > 0)
            }
            __syncthreads();
            const int p = leave_s;
            if (p < 0) break;
            // pivot on (p, q)
            for (int r = tid; r < H; r += kLpThreads) colq[r] = Tb[(int64_t)r * W + q];
            __syncthreads();
            const double inv = 1.0 / colq[p];
            for (int c = tid; c < W; c += kLpThreads) Tb[(int64_t)p * W + c] *= inv;
            __syncthreads();
            for (int k = tid; k < H * W; k += kLpThreads) {
                const int r = k / W;
                if (r == p) continue;
                const int c = k - r * W;
                const double f = colq[r];
                if (f != 0.0) Tb[k] = fma(-f, Tb[(int64_t)p * W + c], Tb[k]);
            }
            if (tid == 0) basis[p] = q;
            __syncthreads();
        }
        if (!done && tid == 0) atomicOr(err, ERRBIT_NOT_CONVERGED);
        // read out: z = sum q = Tb[m][W-1]; v_B = 1 / z
        const double z = Tb[(int64_t)m * W + W - 1];
        const double vB = 1.0 / z;
        for (int j = tid; j < n; j += kLpThreads) y_out[(int64_t)g * n + j] = 0.0;
        __syncthreads();
        for (int r = tid; r < m; r += kLpThreads)
            if (basis[r] < n) y_out[(int64_t)g * n + basis[r]] = Tb[(int64_t)r * W + W - 1] * vB;
        for (int i = tid; i < m; i += kLpThreads) x_out[(int64_t)g * m + i] = Tb[(int64_t)m * W + n + i] * vB;
        if (tid == 0) val_out[g] = vB - shift;
        __syncthreads();
    }
}

}  // namespace

int fp_grid(int32_t n_games, int n_sm) { return n_games < 4 * n_sm ? n_games : 4 * n_sm; }

cudaError_t launch_fictitious_play(const double* P, int32_t G, int32_t m, int32_t n, int32_t stride,
                                   int64_t T, double* x, double* y, double* bounds, int n_sm,
                                   cudaStream_t s) {
    const int ld = n | 1;
    const int64_t bytes = (int64_t)m * ld * 8;
    const int on_chip = bytes <= kSmemLimit ? 1 : 0;
    const size_t dyn = on_chip ? (size_t)bytes : 0;
    cudaError_t e = cudaFuncSetAttribute(fictitious_play_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dyn);
    if (e != cudaSuccess) return e;
    fictitious_play_kernel<<<fp_grid(G, n_sm), kFpThreads, dyn, s>>>(P, G, m, n, stride, T, x, y,
                                                                    bounds, on_chip);
    return cudaGetLastError();
}

cudaError_t launch_aggregate(const double* P, int32_t G, int32_t m, int32_t n, int32_t stride,
                             const double* x, const double* y, double* ay, double* xa, double* val,
                             int n_sm, cudaStream_t s) {
    aggregate_kernel<<<fp_grid(G, n_sm), 256, 0, s>>>(P, G, m, n, stride, x, y, ay, xa, val);
    return cudaGetLastError();
}

int64_t lp_tableau_doubles(int32_t m, int32_t n) { return (int64_t)(m + 1) * (n + m + 1); }

bool lp_on_chip(int32_t m, int32_t n) { return lp_tableau_doubles(m, n) * 8 <= kSmemLimit; }

int lp_grid(int32_t n_games, int n_sm) { return n_games < n_sm ? n_games : n_sm; }

cudaError_t launch_lp_nash(const double* P, int32_t G, int32_t m, int32_t n, int32_t stride,
                           double* x, double* y, double* val, double* scratch, int* err, int n_sm,
                           cudaStream_t s) {
    const int on_chip = lp_on_chip(m, n) ? 1 : 0;
    const size_t dyn = on_chip ? (size_t)lp_tableau_doubles(m, n) * 8 : 0;
    cudaError_t e = cudaFuncSetAttribute(lp_nash_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)dyn);
    if (e != cudaSuccess) return e;
    lp_nash_kernel<<<lp_grid(G, n_sm), kLpThreads, dyn, s>>>(P, G, m, n, stride, x, y, val, scratch,
                                                             on_chip, err);
    return cudaGetLastError();
}

}  // namespace malib

// ---------------------------------------------------------------------------
// C ABI
// ---------------------------------------------------------------------------
using namespace malib;

namespace {

bool dev_ptr(const void* p) {
    if (!p) return false;
    cudaPointerAttributes at;
    if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    return at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged;
}

struct DevSel {
    int prev = -1;
    bool ok = true;
    explicit DevSel(int dev) {
        if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
        ok = cudaSetDevice(dev) == cudaSuccess;
    }
    ~DevSel() {
        if (prev >= 0) cudaSetDevice(prev);
    }
};

int check_table(malib_ctx* ctx, const double* payoff, int32_t G, int32_t m, int32_t n,
                int32_t stride, int32_t max_dim) {
    if (G < 0) return ctx_fail(ctx, MALIB_EINVAL, "n_games < 0");
    if (m < 1 || n < 1 || m > max_dim || n > max_dim)
        return ctx_fail(ctx, m < 1 || n < 1 ? MALIB_EINVAL : MALIB_EUNSUPPORTED,
                        "payoff table dimensions outside 1..limit (see malib.h)");
    if (stride < 1) return ctx_fail(ctx, MALIB_EINVAL, "stride < 1");
    if ((int64_t)G * m * n * stride > ((int64_t)1 << 40))
        return ctx_fail(ctx, MALIB_EINVAL, "payoff table too large");
    if (G > 0 && !dev_ptr(payoff)) return ctx_fail(ctx, MALIB_EINVAL, "payoff must be device memory");
    return MALIB_OK;
}

int launched(malib_ctx* ctx, cudaError_t e, int n_launch) {
    if (e != cudaSuccess) return ctx_fail(ctx, MALIB_ECUDA, cudaGetErrorString(e));
    ctx_count_launches(ctx, n_launch);
    return MALIB_OK;
}

}  // namespace

extern "C" int malib_meta_fictitious_play(malib_ctx* ctx, const double* payoff, int32_t n_games,
                                          int32_t m, int32_t n, int32_t stride, int64_t iters,
                                          double* x_out, double* y_out, double* bounds_out) {
    CtxView v;
    if (!ctx_view(ctx, &v)) return MALIB_EINVAL;
    int r = check_table(ctx, payoff, n_games, m, n, stride, kFpMaxDim);
    if (r != MALIB_OK) return r;
    if (iters < 1) return ctx_fail(ctx, MALIB_EINVAL, "iters must be >= 1");
    if (n_games == 0) return MALIB_OK;
    if (!dev_ptr(x_out) || !dev_ptr(y_out) || !dev_ptr(bounds_out))
        return ctx_fail(ctx, MALIB_EINVAL, "x_out, y_out and bounds_out must be device memory");
    DevSel d(v.device);
    if (!d.ok) return ctx_fail(ctx, MALIB_ECUDA, "cannot select the context's device");
    return launched(ctx, launch_fictitious_play(payoff, n_games, m, n, stride, iters, x_out, y_out,
                                                bounds_out, v.n_sm, v.stream), 1);
}

extern "C" int malib_meta_aggregate(malib_ctx* ctx, const double* payoff, int32_t n_games,
                                    int32_t m, int32_t n, int32_t stride, const double* x,
                                    const double* y, double* row_payoff_out,
                                    double* col_payoff_out, double* value_out) {
    CtxView v;
    if (!ctx_view(ctx, &v)) return MALIB_EINVAL;
    int r = check_table(ctx, payoff, n_games, m, n, stride, 1 << 20);
    if (r != MALIB_OK) return r;
    if (n_games == 0) return MALIB_OK;
    if (!dev_ptr(x) || !dev_ptr(y) || !dev_ptr(row_payoff_out) || !dev_ptr(col_payoff_out) ||
        !dev_ptr(value_out))
        return ctx_fail(ctx, MALIB_EINVAL, "mixtures and outputs must be device memory");
    DevSel d(v.device);
    if (!d.ok) return ctx_fail(ctx, MALIB_ECUDA, "cannot select the context's device");
    return launched(ctx, launch_aggregate(payoff, n_games, m, n, stride, x, y, row_payoff_out,
                                          col_payoff_out, value_out, v.n_sm, v.stream), 1);
}

extern "C" int malib_meta_lp_nash(malib_ctx* ctx, const double* payoff, int32_t n_games, int32_t m,
                                  int32_t n, int32_t stride, double* x_out, double* y_out,
                                  double* value_out) {
    CtxView v;
    if (!ctx_view(ctx, &v)) return MALIB_EINVAL;
    int r = check_table(ctx, payoff, n_games, m, n, stride, 512);
    if (r != MALIB_OK) return r;
    if (n_games == 0) return MALIB_OK;
    if (!dev_ptr(x_out) || !dev_ptr(y_out) || !dev_ptr(value_out))
        return ctx_fail(ctx, MALIB_EINVAL, "x_out, y_out and value_out must be device memory");
    DevSel d(v.device);
    if (!d.ok) return ctx_fail(ctx, MALIB_ECUDA, "cannot select the context's device");
    double* scratch = nullptr;
    if (!lp_on_chip(m, n)) {
        void* p = nullptr;
        r = ctx_scratch(ctx, (int64_t)lp_grid(n_games, v.n_sm) * lp_tableau_doubles(m, n) * 8, &p);
        if (r != MALIB_OK) return r;
        scratch = static_cast<double*>(p);
    }
    return launched(ctx, launch_lp_nash(payoff, n_games, m, n, stride, x_out, y_out, value_out,
                                        scratch, v.err, v.n_sm, v.stream), 1);
}
