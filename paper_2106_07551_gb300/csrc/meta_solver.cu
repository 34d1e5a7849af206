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

// Order-preserving integer key of a finite double (larger double, larger
// key), and its inverse. The comparisons of a play run on these keys: fp64
// arithmetic is a narrow pipe on this part, integer compares and shuffles are
// not. The cumulative payoffs start at +0.0 and every sum with +0.0 is +0.0,
// so -0.0 never occurs and key equality is value equality.
__device__ __forceinline__ long long okey(double v) {
    const long long b = __double_as_longlong(v);
    return b >= 0 ? b : b ^ 0x7fffffffffffffffll;
}
__device__ __forceinline__ double okey_inv(long long k) {
    return __longlong_as_double(k >= 0 ? k : k ^ 0x7fffffffffffffffll);
}

struct Cand {
    long long k;      // key to maximise; kNone for "no candidate"
    int i;            // index; ties go to the lower one
};
constexpr long long kNone = (long long)0x8000000000000000ull;   // below every finite key

// Branch-free: b replaces a when its key is larger, or equal with a lower index.
__device__ __forceinline__ Cand pick(Cand a, Cand b) {
    const bool take = (b.k > a.k) | ((b.k == a.k) & (b.i < a.i));
    return Cand{take ? b.k : a.k, take ? b.i : a.i};
}

template <int kSteps>
__device__ __forceinline__ Cand warp_pick(Cand a) {
#pragma unroll
    for (int s = 0; s < kSteps; ++s) {
        const int o = 1 << s;                   // butterfly over lane bits 0 .. kSteps-1
        Cand b;
        b.k = __shfl_xor_sync(0xffffffffu, a.k, o);
        b.i = __shfl_xor_sync(0xffffffffu, a.i, o);
        a = pick(a, b);
    }
    return a;
}

// Simultaneous fictitious play: both play policy 0 first; then each plays the
// first best response to the other's plays so far. u_row[i] = sum over plays
// of A[i][j_s] and u_col[j] = sum of A[i_s][j] are fp64 sums in play order,
// held in registers with the play counts (thread t owns rows and columns t,
// t + blockDim, ...). One CTA barrier per play: every warp publishes its best
// row and column into a buffer selected by the play's parity, and after the
// barrier every warp reduces the published candidates itself, so all threads
// know the next plays. The column player's argmin is the argmax of the
// negated key.
template <bool kOnChip>
__global__ void __launch_bounds__(kFpThreads) fictitious_play_kernel(
    const double* __restrict__ P, int32_t n_games, int32_t m, int32_t n, int32_t stride,
    int64_t T, double* __restrict__ x_out, double* __restrict__ y_out,
    double* __restrict__ bounds_out) {
    extern __shared__ double sA[];              // [m][ld] when on chip
    __shared__ Cand red[2][2][8];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int nt = blockDim.x;
    const int ld = n | 1;                       // odd row stride: column reads hit distinct banks

    for (int g = blockIdx.x; g < n_games; g += gridDim.x) {
        const double* Pg = P + (int64_t)g * m * n * stride;
        __syncthreads();                        // the previous game's readers are done
        if (kOnChip) {
            for (int k = tid; k < m * n; k += nt) {
                const int i = k / n, j = k - i * n;
                sA[i * ld + j] = Pg[(int64_t)k * stride];
            }
        }
        if (tid < 32) {
            const Cand none{kNone, 0x7fffffff};
            (&red[0][0][0])[tid] = none;
        }
        __syncthreads();
        auto a_at = [&](int i, int j) -> double {
            return kOnChip ? sA[i * ld + j] : __ldg(Pg + ((int64_t)i * n + j) * stride);
        };
        double ur[kFpPer], uc[kFpPer];
        long long cr[kFpPer], cc[kFpPer];
#pragma unroll
        for (int k = 0; k < kFpPer; ++k) { ur[k] = 0.0; uc[k] = 0.0; cr[k] = 0; cc[k] = 0; }
        int it = 0, jt = 0;
        Cand top{kNone, 0x7fffffff}, bot{kNone, 0x7fffffff};
        for (int64_t t = 0; t < T; ++t) {
            const int par = (int)(t & 1);
            Cand br{kNone, 0x7fffffff}, bc{kNone, 0x7fffffff};
#pragma unroll
            for (int k = 0; k < kFpPer; ++k) {
                const int i = tid + k * nt;
                if (i < m) {
                    cr[k] += (i == it);
                    ur[k] += a_at(i, jt);
                    br = pick(br, Cand{okey(ur[k]), i});
                }
                if (i < n) {
                    cc[k] += (i == jt);
                    uc[k] += a_at(it, i);
                    bc = pick(bc, Cand{-okey(uc[k]), i});
                }
            }
            br = warp_pick<5>(br);
            bc = warp_pick<5>(bc);
            if (lane == 0) { red[par][0][warp] = br; red[par][1][warp] = bc; }
            __syncthreads();
            // at most 8 published candidates (unused entries hold "none"); every
            // group of 8 lanes holds all of them, reduced over lane bits 0..2
            top = warp_pick<3>(red[par][0][lane & 7]);
            bot = warp_pick<3>(red[par][1][lane & 7]);
            it = top.i;
            jt = bot.i;
        }
        const double Td = (double)T;
#pragma unroll
        for (int k = 0; k < kFpPer; ++k) {
            const int i = tid + k * nt;
            if (i < m) x_out[(int64_t)g * m + i] = (double)cr[k] / Td;
            if (i < n) y_out[(int64_t)g * n + i] = (double)cc[k] / Td;
        }
        if (tid == 0) {
            bounds_out[2 * g] = okey_inv(-bot.k) / Td;     // min_j (x^T A)_j
            bounds_out[2 * g + 1] = okey_inv(top.k) / Td;  // max_i (A y)_i
        }
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
// Tableau rows 0..m-1: [B | I | 1]; row m: [-1 ... -1 | 0 | 0].
// Entering column: the most negative reduced cost (Dantzig); after 2 (m + n)
// consecutive degenerate pivots the rule switches for good to Bland's (lowest
// index with a negative reduced cost), which cannot cycle. Leaving row: the
// minimum ratio, ties to the lowest basic variable index. A pivot limit (at
// most that many pivots; optimality is still recognised after the last one)
// guards regardless. Comparisons run on the integer keys above; the tableau
// arithmetic is fp64.
// ---------------------------------------------------------------------------
constexpr int kLpThreads = 512;
constexpr int kLpWarps = kLpThreads / 32;

// Reduction of one candidate per thread to the CTA's best (all threads get it).
__device__ __forceinline__ Cand cta_pick(Cand c, Cand* red) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    c = warp_pick<5>(c);
    __syncthreads();                             // red's previous readers are done
    if (lane == 0) red[warp] = c;
    __syncthreads();
    return warp_pick<4>(red[lane & 15]);
}

__global__ void __launch_bounds__(kLpThreads) lp_nash_kernel(
    const double* __restrict__ P, int32_t n_games, int32_t m, int32_t n, int32_t stride,
    double* __restrict__ x_out, double* __restrict__ y_out, double* __restrict__ val_out,
    double* __restrict__ gscratch, int32_t on_chip, int32_t pivot_limit, int* __restrict__ err) {
    extern __shared__ double smem_tab[];
    __shared__ double colq[1024 + 1];
    __shared__ int basis[1024];
    __shared__ Cand red[kLpWarps];
    const int tid = threadIdx.x;
    const int W = n + m + 1;                     // tableau width; column W-1 is the right side
    const int H = m + 1;                         // rows; row m is the objective
    const Cand none{kNone, 0x7fffffff};
    const double eps = 1e-12;
    const long long k_neg_eps = okey(-eps);

    for (int g = blockIdx.x; g < n_games; g += gridDim.x) {
        double* Tb = on_chip ? smem_tab : gscratch + (int64_t)blockIdx.x * H * W;
        const double* Pg = P + (int64_t)g * m * n * stride;
        Cand lo = none;                          // min(A): the largest negated key
        for (int k = tid; k < m * n; k += kLpThreads)
            lo = pick(lo, Cand{-okey(Pg[(int64_t)k * stride]), k});
        lo = cta_pick(lo, red);
        const double shift = 1.0 - okey_inv(-lo.k);
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

        const int max_pivots = pivot_limit > 0 ? pivot_limit : 50 * (m + n) + 1000;
        bool done = false, bland = false;
        int degenerate = 0;
        for (int piv = 0;; ++piv) {
            // entering column
            Cand ce = none;
            for (int c = tid; c < n + m; c += kLpThreads) {
                const long long k = okey(Tb[(int64_t)m * W + c]);
                if (k < k_neg_eps) ce = pick(ce, Cand{bland ? 0ll : -k, c});
            }
            ce = cta_pick(ce, red);
            if (ce.k == kNone) { done = true; break; }
            if (piv == max_pivots) break;        // another pivot is needed: limit reached
            const int q = ce.i;
            // leaving row: minimum ratio (ratios are >= 0), ties to the lowest
            // basic index; the candidate index packs (basic index, row)
            Cand cl = none;
            for (int r = tid; r < m; r += kLpThreads) {
                const double a = Tb[(int64_t)r * W + q];
                if (a > eps) {
                    const double ratio = Tb[(int64_t)r * W + W - 1] / a;
                    cl = pick(cl, Cand{-okey(ratio), basis[r] * 1024 + r});
                }
            }
            cl = cta_pick(cl, red);
            if (cl.k == kNone) break;            // unbounded: cannot happen with B > 0
            const int p = cl.i & 1023;
            degenerate = (okey_inv(-cl.k) == 0.0) ? degenerate + 1 : 0;
            if (degenerate > 2 * (m + n)) bland = true;
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
    const bool on_chip = bytes <= kSmemLimit;
    const size_t dyn = on_chip ? (size_t)bytes : 0;
    // one thread per row and column up to 256 of them (fewer warps, cheaper
    // barriers), else 256 threads with up to kFpPer rows / columns each
    const int mx = m > n ? m : n;
    const int threads = mx <= kFpThreads ? ((mx + 31) / 32) * 32 : kFpThreads;
    auto kern = on_chip ? fictitious_play_kernel<true> : fictitious_play_kernel<false>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dyn);
    if (e != cudaSuccess) return e;
    kern<<<fp_grid(G, n_sm), threads, dyn, s>>>(P, G, m, n, stride, T, x, y, bounds);
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
                           double* x, double* y, double* val, double* scratch, int32_t pivot_limit,
                           int* err, int n_sm, cudaStream_t s) {
    const int on_chip = lp_on_chip(m, n) ? 1 : 0;
    const size_t dyn = on_chip ? (size_t)lp_tableau_doubles(m, n) * 8 : 0;
    cudaError_t e = cudaFuncSetAttribute(lp_nash_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)dyn);
    if (e != cudaSuccess) return e;
    lp_nash_kernel<<<lp_grid(G, n_sm), kLpThreads, dyn, s>>>(P, G, m, n, stride, x, y, val, scratch,
                                                             on_chip, pivot_limit, err);
    return cudaGetLastError();
}

}  // namespace malib

// ---------------------------------------------------------------------------
// C ABI
// ---------------------------------------------------------------------------
using namespace malib;

namespace {

// Device memory of the context's own device.
bool dev_ptr(int device, const void* p) { return p && ptr_where(p, device) == kPtrHere; }

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

int check_table(malib_ctx* ctx, int device, const double* payoff, int32_t G, int32_t m, int32_t n,
                int32_t stride, int32_t max_dim) {
    if (G < 0) return ctx_fail(ctx, MALIB_EINVAL, "n_games < 0");
    if (m < 1 || n < 1 || m > max_dim || n > max_dim)
        return ctx_fail(ctx, m < 1 || n < 1 ? MALIB_EINVAL : MALIB_EUNSUPPORTED,
                        "payoff table dimensions outside 1..limit (see malib.h)");
    if (stride < 1) return ctx_fail(ctx, MALIB_EINVAL, "stride < 1");
    if ((int64_t)G * m * n * stride > ((int64_t)1 << 40))
        return ctx_fail(ctx, MALIB_EINVAL, "payoff table too large");
    if (G > 0 && !dev_ptr(device, payoff)) return ctx_fail(ctx, MALIB_EINVAL, "payoff must be device memory of the context's device");
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
    int r = check_table(ctx, v.device, payoff, n_games, m, n, stride, kFpMaxDim);
    if (r != MALIB_OK) return r;
    if (iters < 1) return ctx_fail(ctx, MALIB_EINVAL, "iters must be >= 1");
    if (n_games == 0) return MALIB_OK;
    if (!dev_ptr(v.device, x_out) || !dev_ptr(v.device, y_out) || !dev_ptr(v.device, bounds_out))
        return ctx_fail(ctx, MALIB_EINVAL, "x_out, y_out and bounds_out must be device memory of the context's device");
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
    int r = check_table(ctx, v.device, payoff, n_games, m, n, stride, 1 << 20);
    if (r != MALIB_OK) return r;
    if (n_games == 0) return MALIB_OK;
    if (!dev_ptr(v.device, x) || !dev_ptr(v.device, y) || !dev_ptr(v.device, row_payoff_out) ||
        !dev_ptr(v.device, col_payoff_out) || !dev_ptr(v.device, value_out))
        return ctx_fail(ctx, MALIB_EINVAL, "mixtures and outputs must be device memory of the context's device");
    DevSel d(v.device);
    if (!d.ok) return ctx_fail(ctx, MALIB_ECUDA, "cannot select the context's device");
    return launched(ctx, launch_aggregate(payoff, n_games, m, n, stride, x, y, row_payoff_out,
                                          col_payoff_out, value_out, v.n_sm, v.stream), 1);
}

extern "C" int malib_meta_lp_nash_ex(malib_ctx* ctx, const double* payoff, int32_t n_games,
                                     int32_t m, int32_t n, int32_t stride, int32_t max_pivots,
                                     double* x_out, double* y_out, double* value_out) {
    CtxView v;
    if (!ctx_view(ctx, &v)) return MALIB_EINVAL;
    int r = check_table(ctx, v.device, payoff, n_games, m, n, stride, 512);
    if (r != MALIB_OK) return r;
    if (max_pivots < 0) return ctx_fail(ctx, MALIB_EINVAL, "max_pivots < 0");
    if (n_games == 0) return MALIB_OK;
    if (!dev_ptr(v.device, x_out) || !dev_ptr(v.device, y_out) || !dev_ptr(v.device, value_out))
        return ctx_fail(ctx, MALIB_EINVAL, "x_out, y_out and value_out must be device memory of the context's device");
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
                                        scratch, max_pivots, v.err, v.n_sm, v.stream), 1);
}

extern "C" int malib_meta_lp_nash(malib_ctx* ctx, const double* payoff, int32_t n_games, int32_t m,
                                  int32_t n, int32_t stride, double* x_out, double* y_out,
                                  double* value_out) {
    return malib_meta_lp_nash_ex(ctx, payoff, n_games, m, n, stride, 0, x_out, y_out, value_out);
}
