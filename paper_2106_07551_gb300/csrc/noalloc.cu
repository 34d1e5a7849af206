// Payoff-table evaluation that allocates no device memory.
//
// Some callers cannot allocate device memory at the moment they need a
// payoff table: a caller whose framework has already reserved the GPU's memory
// in its own caching pool (a cudaMalloc would then fail or fragment it), a
// caller running a latency-critical loop in which cudaMalloc / cudaFree would
// synchronise the whole device and stall other streams, or an embedding whose
// rules forbid allocations after start-up. malib_eval_payoff_noalloc serves
// them: it runs the same evaluation kernels as malib_eval_payoff, but its
// scratch (the per-pair payoff sums and the decision counter) lives in the
// file-scope device array below instead of context-owned memory grown with
// cudaMallocAsync, and it stages nothing (pair table and output must already
// be device buffers). The scratch also holds the per-pair hand counters from
// which the fp32 Leduc kernel's CTAs claim hands.
//
// The array has room for kNoAllocMaxPairs pairs: (3 * 8192 + 1) x 8 bytes
// (sums, decision counter, hand counters), 192 KiB + 8 B, held by every GPU
// that loads the library until the process exits. Every call shares it and it keeps the previous call's contents, so
// each call clears it first; calls that overlap on the GPU (two streams, or two
// contexts on one device) race on it and must be serialised by the caller.
#include <cstdint>
#include <mutex>

#include "internal.h"
#include "malib.h"

namespace malib {

namespace {

constexpr int32_t kNoAllocMaxPairs = 8192;
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned long long g_noalloc_scratch[3 * kNoAllocMaxPairs + 1];

std::mutex g_mu;
unsigned long long* g_scratch_addr[kMaxDevices] = {};

// Device address of g_noalloc_scratch on the current device. In host code the
// array's name only stands in for it; the address comes from
// cudaGetSymbolAddress, looked up once per device (with that device current).
cudaError_t scratch_address(int device, unsigned long long** out) {
    std::lock_guard<std::mutex> lock(g_mu);
    if (!g_scratch_addr[device]) {
        void* p = nullptr;
        const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess) return e;
        g_scratch_addr[device] = static_cast<unsigned long long*>(p);
    }
    *out = g_scratch_addr[device];
    return cudaSuccess;
}

}  // namespace

}  // namespace malib

using namespace malib;

extern "C" int malib_eval_payoff_noalloc(malib_ctx* ctx, const int32_t* pair_ids, int32_t n_pairs,
                                         int64_t n_episodes, uint64_t seed, double* payoff_out) {
    CtxView v;
    if (!ctx_view(ctx, &v)) return MALIB_EINVAL;
    if (!v.has_pop) return ctx_fail(ctx, MALIB_ESTATE, "no population loaded");
    if (v.env_kind != MALIB_ENV_KUHN && v.env_kind != MALIB_ENV_LEDUC)
        return ctx_fail(ctx, MALIB_ESTATE, "payoff evaluation needs a Kuhn or Leduc population");
    if (v.env_kind == MALIB_ENV_LEDUC &&
        (v.pol_dtype != MALIB_F32 || v.dims[1] != v.dims[2] || !leduc_f32_supported(v.dims[1])))
        return ctx_fail(ctx, MALIB_EUNSUPPORTED, "no fp32 Leduc kernel for this policy shape");
    if (n_pairs < 0) return ctx_fail(ctx, MALIB_EINVAL, "n_pairs < 0");
    if (n_pairs > kNoAllocMaxPairs)
        return ctx_fail(ctx, MALIB_EINVAL,
                        "malib_eval_payoff_noalloc takes at most 8192 pairs per call "
                        "(its fixed scratch holds 8192 payoff entries)");
    if (n_pairs == 0) return MALIB_OK;
    if (n_episodes < 1) return ctx_fail(ctx, MALIB_EINVAL, "n_episodes must be >= 1");
    if (n_episodes > ((int64_t)1 << 40) / n_pairs)
        return ctx_fail(ctx, MALIB_EINVAL, "n_pairs * n_episodes too large");
    if (!pair_ids || !payoff_out) return ctx_fail(ctx, MALIB_EINVAL, "pair_ids or payoff_out is NULL");
    if (!v.tables_uploaded)
        return ctx_fail(ctx, MALIB_ESTATE, "population tables are not on the device");

    int prev = -1;
    if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
    if (cudaSetDevice(v.device) != cudaSuccess || v.device >= kMaxDevices) {
        if (prev >= 0) cudaSetDevice(prev);
        return ctx_fail(ctx, MALIB_ECUDA, "cannot select the context's device");
    }
    int code = MALIB_OK;
    unsigned long long* scratch = nullptr;
    cudaError_t e;
    if (ptr_where(pair_ids, v.device) != kPtrHere || ptr_where(payoff_out, v.device) != kPtrHere) {
        code = ctx_fail(ctx, MALIB_EINVAL,
                        "malib_eval_payoff_noalloc needs pair_ids and payoff_out in device memory "
                        "of the context's device (host buffers would need a staging allocation)");
    } else if ((e = scratch_address(v.device, &scratch)) != cudaSuccess) {
        code = ctx_fail(ctx, MALIB_ECUDA, cudaGetErrorString(e));
    } else {
        EvalArgs a{};
        a.arena = v.arena;
        a.pol_offset = v.pol_offset;
        a.pol_seat = v.pol_seat;
        a.n_pol = v.n_pol;
        a.err = v.err;
        a.pairs = pair_ids;
        a.n_pairs = n_pairs;
        a.n_episodes = n_episodes;
        a.seed = seed;
        a.acc = scratch;
        a.n_dec = scratch + 2 * (int64_t)n_pairs;
        a.work = scratch + 2 * (int64_t)n_pairs + 1;
        if ((e = launch_zero_u64(scratch, 3 * (int64_t)n_pairs + 1, v.stream)) == cudaSuccess)
            e = v.env_kind == MALIB_ENV_KUHN ? launch_kuhn_eval(a, v.n_sm, v.stream)
                                             : launch_leduc_eval_f32(a, v.dims[1], v.n_sm, v.stream);
        if (e == cudaSuccess) e = launch_finalize(scratch, n_pairs, n_episodes, payoff_out, v.stream);
        if (e != cudaSuccess) code = ctx_fail(ctx, MALIB_ECUDA, cudaGetErrorString(e));
        else ctx_count_launches(ctx, 3);
    }
    if (prev >= 0) cudaSetDevice(prev);
    return code;
}
