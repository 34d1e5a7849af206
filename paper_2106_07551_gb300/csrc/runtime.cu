// Host runtime behind the C ABI of include/malib.h: context, population arena,
// argument validation, pointer classification, launches, deferred device
// errors and measurement hooks.
#include <algorithm>
#include <cstdarg>
#include <cstdio>
#include <cmath>
#include <cstring>
#include <mutex>
#include <string>
#include <utility>
#include <vector>

#include "internal.h"
#include "malib.h"
#include "tc_common.cuh"

using namespace malib;

namespace {

struct PolicyRec {
    int kind, dtype, seat;
    int dims[4];
    int64_t offset;   // floats into the arena
};

}  // namespace

struct malib_ctx {
    int device = 0;
    cudaStream_t stream = nullptr;
    int n_sm = 1;
    std::string err;

    bool has_pop = false;
    malib_env_spec spec{};
    int pol_kind = 0, pol_dtype = 0;
    int dims[4] = {0, 0, 0, 0};
    bool tc_layout = false;            // bf16 tensor-core images in the arena
    std::vector<PolicyRec> pols;
    float* arena = nullptr;
    int64_t arena_cap = 0;             // floats
    int64_t arena_used = 0;            // floats
    float* d_stage = nullptr;          // plain parameters of a load, before conversion
    int64_t stage_cap = 0;
    ConvJob* d_jobs = nullptr;
    int64_t jobs_cap = 0;
    int64_t* d_off = nullptr;
    int32_t* d_seat = nullptr;
    int64_t tbl_cap = 0;
    int64_t seat_cap = 0;
    bool tables_dirty = false;

    unsigned long long* acc = nullptr;
    int64_t acc_cap = 0;
    int64_t last_pairs = -1;           // n_pairs of the last Monte-Carlo evaluation
    int* d_err = nullptr;
    int32_t* d_pairs = nullptr;
    int64_t pairs_cap = 0;
    double* d_out = nullptr;
    int64_t out_cap = 0;
    uint8_t* scratch = nullptr;        // solver work space (LP tableaus that do not fit on chip)
    int64_t scratch_cap = 0;
    uint8_t* lwork = nullptr;          // tensor-core Leduc evaluation: hand states and queues
    int64_t lwork_cap = 0;
    uint8_t* learn_work = nullptr;     // policy-gradient step: slots, returns, partial gradients
    int64_t learn_work_cap = 0;
    float* learn_grad = nullptr;       // the gradient when the caller's buffer is host memory
    int64_t learn_grad_cap = 0;

    int64_t launches = 0;
    bool timing = false;
    std::vector<std::pair<cudaEvent_t, cudaEvent_t>> events;
    double timed_ms = 0.0;
    int64_t timed_n = 0;
};

namespace {

thread_local std::string g_create_err;

struct DeviceGuard {
    int prev = -1;
    bool ok = true;
    explicit DeviceGuard(int dev) {
        if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
        ok = cudaSetDevice(dev) == cudaSuccess;
    }
    ~DeviceGuard() {
        if (prev >= 0) cudaSetDevice(prev);
    }
};

int fail(malib_ctx* c, int code, const char* fmt, ...) __attribute__((format(printf, 3, 4)));
int fail(malib_ctx* c, int code, const char* fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    if (c) c->err = buf;
    else g_create_err = buf;
    return code;
}

int cuda_fail(malib_ctx* c, cudaError_t e, const char* what) {
    return fail(c, e == cudaErrorMemoryAllocation ? MALIB_ENOMEM : MALIB_ECUDA, "%s: %s", what,
                cudaGetErrorString(e));
}

#define CK(call, what)                                 \
    do {                                               \
        cudaError_t e_ = (call);                       \
        if (e_ != cudaSuccess) return cuda_fail(c, e_, what); \
    } while (0)

// Device memory of the context's own device (or managed memory).
bool is_device_ptr(const malib_ctx* c, const void* p) { return ptr_where(p, c->device) == kPtrHere; }

template <class T>
int ensure(malib_ctx* c, T*& p, int64_t& cap, int64_t need, const char* what) {
    if (need <= cap) return MALIB_OK;
    int64_t n = cap > 0 ? cap : 64;
    while (n < need) n *= 2;
    if (p) cudaFreeAsync(p, c->stream);
    p = nullptr;
    cap = 0;
    CK(cudaMallocAsync((void**)&p, (size_t)n * sizeof(T), c->stream), what);
    cap = n;
    return MALIB_OK;
}

int64_t mlp_param_floats(const int* d) {
    return (int64_t)d[1] * d[0] + d[1] + (int64_t)d[2] * d[1] + d[2] + (int64_t)d[3] * d[2] + d[3];
}

int check_spec(malib_ctx* c, const malib_env_spec* s) {
    if (!s) return fail(c, MALIB_EINVAL, "env spec is NULL");
    switch (s->env_kind) {
        case MALIB_ENV_KUHN:
            if (s->n_agents != 2 || s->obs_dim != 0 || s->n_actions != 2)
                return fail(c, MALIB_EINVAL, "Kuhn spec needs n_agents 2, obs_dim 0, n_actions 2");
            break;
        case MALIB_ENV_LEDUC:
            if (s->n_agents != 2 || s->obs_dim != 17 || s->n_actions != 3)
                return fail(c, MALIB_EINVAL, "Leduc spec needs n_agents 2, obs_dim 17, n_actions 3");
            break;
        case MALIB_ENV_SPREAD: {
            const int n = s->n_agents;
            if (n < 2 || n > kMaxAgents || s->n_landmarks != n || s->n_actions != 5)
                return fail(c, MALIB_EINVAL,
                            "spread spec needs 2 <= n_agents == n_landmarks <= 16 and n_actions 5");
            if (s->obs_dim < 4 + 2 * n + 2 * (n - 1))
                return fail(c, MALIB_EINVAL, "spread obs_dim %d below the %d features", s->obs_dim,
                            4 + 2 * n + 2 * (n - 1));
            if (s->episode_len < 1) return fail(c, MALIB_EINVAL, "episode_len must be >= 1");
            break;
        }
        case MALIB_ENV_ADVERSARY:
            if (s->n_agents != 3 || s->n_landmarks != 2 || s->obs_dim != 14 || s->n_actions != 5)
                return fail(c, MALIB_EINVAL,
                            "adversary spec needs n_agents 3, n_landmarks 2, obs_dim 14, n_actions 5");
            if (s->episode_len < 1) return fail(c, MALIB_EINVAL, "episode_len must be >= 1");
            break;
        case MALIB_ENV_SPEAKER_LISTENER:
            if (s->n_agents != 2 || s->n_landmarks != 3 || s->obs_dim != 11 || s->n_actions != 5)
                return fail(c, MALIB_EINVAL,
                            "speaker-listener spec needs n_agents 2, n_landmarks 3, obs_dim 11, n_actions 5");
            if (s->episode_len < 1) return fail(c, MALIB_EINVAL, "episode_len must be >= 1");
            break;
        case MALIB_ENV_PUSH:
            if (s->n_agents != 2 || s->n_landmarks != 1 || s->obs_dim != 8 || s->n_actions != 5)
                return fail(c, MALIB_EINVAL, "push spec needs n_agents 2, n_landmarks 1, obs_dim 8, n_actions 5");
            if (s->episode_len < 1) return fail(c, MALIB_EINVAL, "episode_len must be >= 1");
            break;
        case MALIB_ENV_REFERENCE:
            if (s->n_agents != 2 || s->n_landmarks != 3 || s->obs_dim != 14 || s->n_actions != 15)
                return fail(c, MALIB_EINVAL, "reference spec needs n_agents 2, n_landmarks 3, obs_dim 14, n_actions 15");
            if (s->episode_len < 1) return fail(c, MALIB_EINVAL, "episode_len must be >= 1");
            break;
        case MALIB_ENV_TAG:
            if (s->n_agents != 4 || s->n_landmarks != 2 || s->obs_dim != 16 || s->n_actions != 5)
                return fail(c, MALIB_EINVAL, "tag spec needs n_agents 4, n_landmarks 2, obs_dim 16, n_actions 5");
            if (s->episode_len < 1) return fail(c, MALIB_EINVAL, "episode_len must be >= 1");
            break;
        default:
            return fail(c, MALIB_EINVAL, "unknown env_kind %d", s->env_kind);
    }
    if (s->flags & ~(MALIB_DUMP_LOGITS | MALIB_EXACT_EXPECTATION | MALIB_SPREAD_LOCAL_RATIO | MALIB_SPREAD_CONTACT))
        return fail(c, MALIB_EINVAL, "unknown flags 0x%x", s->flags);
    if ((s->flags & MALIB_SPREAD_CONTACT) && s->env_kind != MALIB_ENV_SPREAD)
        return fail(c, MALIB_EINVAL, "MALIB_SPREAD_CONTACT applies to SPREAD only");
    if (s->flags & MALIB_SPREAD_LOCAL_RATIO) {
        if (s->env_kind != MALIB_ENV_SPREAD && s->env_kind != MALIB_ENV_REFERENCE)
            return fail(c, MALIB_EINVAL, "MALIB_SPREAD_LOCAL_RATIO applies to SPREAD and REFERENCE only");
        if (!(s->local_ratio >= 0.0f && s->local_ratio <= 1.0f))
            return fail(c, MALIB_EINVAL, "local_ratio must lie in [0, 1]");
    }
    return MALIB_OK;
}

bool same_env(const malib_env_spec& a, const malib_env_spec& b) {
    return a.env_kind == b.env_kind && a.n_agents == b.n_agents &&
           a.n_landmarks == b.n_landmarks && a.obs_dim == b.obs_dim && a.n_actions == b.n_actions;
}

int upload_tables(malib_ctx* c) {
    if (!c->tables_dirty) return MALIB_OK;
    const int64_t n = (int64_t)c->pols.size();
    int r;
    if ((r = ensure(c, c->d_off, c->tbl_cap, std::max<int64_t>(n, 1), "policy table")) != MALIB_OK)
        return r;
    if ((r = ensure(c, c->d_seat, c->seat_cap, std::max<int64_t>(n, 1), "seat table")) != MALIB_OK)
        return r;
    std::vector<int64_t> off(n);
    std::vector<int32_t> seat(n);
    for (int64_t i = 0; i < n; ++i) { off[i] = c->pols[i].offset; seat[i] = c->pols[i].seat; }
    CK(cudaMemcpyAsync(c->d_off, off.data(), n * 8, cudaMemcpyHostToDevice, c->stream), "upload");
    CK(cudaMemcpyAsync(c->d_seat, seat.data(), n * 4, cudaMemcpyHostToDevice, c->stream), "upload");
    CK(cudaStreamSynchronize(c->stream), "upload");
    c->tables_dirty = false;
    return MALIB_OK;
}

// The conversion of a policy's parameters into its kernel image: kind, flags
// and image size (words).
void conv_job(int env_kind, int kind, int dtype, const int* dims, ConvJob* jb) {
    std::memcpy(jb->dims, dims, sizeof jb->dims);
    jb->flags = 0;
    if (kind == MALIB_POL_TABULAR) {
        jb->kind = kConvTable;
        jb->size = 8;
    } else if (dtype == MALIB_BF16 && tc_image_shape(dims)) {
        const bool fold = leduc_tc_fold(env_kind, dims[0]);
        jb->kind = kConvTc;
        jb->flags = fold ? kConvFold : 0;
        jb->size = tc_image_bytes(fold ? dims[0] - 1 : dims[0]) / 4;
    } else {
        jb->kind = kConvF32;
        jb->flags = dtype == MALIB_BF16 ? kConvRound : 0;   // bf16 weights, fp32 biases
        jb->size = ((int64_t)dims[0] * dims[1] + dims[1] + (int64_t)dims[1] * dims[2] + dims[2] +
                    (int64_t)dims[3] * dims[2] + dims[3] + 3) / 4 * 4;
    }
}

int stage_pairs(malib_ctx* c, const int32_t* pair_ids, int64_t n_ints, int width, bool poker,
                const int32_t** dev_pairs) {
    const int where = ptr_where(pair_ids, c->device);
    if (where == kPtrOther)
        return fail(c, MALIB_EINVAL, "pair_ids lives on another device than the context's");
    if (where == kPtrHere) {
        *dev_pairs = pair_ids;      // validated by the kernels
        return MALIB_OK;
    }
    const int64_t n_pol = (int64_t)c->pols.size();
    for (int64_t i = 0; i < n_ints; ++i) {
        const int32_t id = pair_ids[i];
        if (id < 0 || id >= n_pol)
            return fail(c, MALIB_EINVAL, "pair_ids[%lld] = %d is not a policy id (population %lld)",
                        (long long)i, id, (long long)n_pol);
        if (poker) {
            const int want = (int)(i % width);
            const int s = c->pols[id].seat;
            if (s != -1 && s != want)
                return fail(c, MALIB_EINVAL, "policy %d belongs to seat %d, used for seat %d", id, s,
                            want);
        }
    }
    int r;
    if ((r = ensure(c, c->d_pairs, c->pairs_cap, std::max<int64_t>(n_ints, 1), "pair staging")) !=
        MALIB_OK)
        return r;
    CK(cudaMemcpyAsync(c->d_pairs, pair_ids, n_ints * 4, cudaMemcpyHostToDevice, c->stream),
       "pair upload");
    *dev_pairs = c->d_pairs;
    return MALIB_OK;
}

int read_device_errors(malib_ctx* c) {
    int h = 0;
    CK(cudaMemcpyAsync(&h, c->d_err, 4, cudaMemcpyDeviceToHost, c->stream), "error flag");
    CK(cudaStreamSynchronize(c->stream), "sync");
    if (h) {
        CK(cudaMemsetAsync(c->d_err, 0, 4, c->stream), "error flag");
        if (h & ERRBIT_TIMEOUT)
            return fail(c, MALIB_ETIMEOUT, "a bounded device wait expired");
        if (h & ERRBIT_BAD_PAIR)
            return fail(c, MALIB_EINVAL, "a device pair table held an invalid policy id or seat");
        if (h & ERRBIT_NOT_CONVERGED)
            return fail(c, MALIB_ENOTCONVERGED, "the LP solver reached its pivot limit");
    }
    return MALIB_OK;
}

void time_begin(malib_ctx* c, cudaEvent_t* a, cudaEvent_t* b) {
    *a = *b = nullptr;
    if (!c->timing) return;
    if (cudaEventCreate(a) != cudaSuccess || cudaEventCreate(b) != cudaSuccess) {
        cudaGetLastError();
        *a = *b = nullptr;
        return;
    }
    cudaEventRecord(*a, c->stream);
}

void time_end(malib_ctx* c, cudaEvent_t a, cudaEvent_t b) {
    if (!a) return;
    cudaEventRecord(b, c->stream);
    c->events.emplace_back(a, b);
}

EvalArgs eval_args(malib_ctx* c) {
    EvalArgs a{};
    a.arena = c->arena;
    a.pol_offset = c->d_off;
    a.pol_seat = c->d_seat;
    a.n_pol = (int32_t)c->pols.size();
    a.err = c->d_err;
    return a;
}

}  // namespace

namespace malib {

int ptr_where(const void* p, int device) {
    cudaPointerAttributes at;
    if (!p || cudaPointerGetAttributes(&at, p) != cudaSuccess) {
        cudaGetLastError();
        return kPtrHost;
    }
    if (at.type == cudaMemoryTypeManaged) return kPtrHere;
    if (at.type == cudaMemoryTypeDevice) return at.device == device ? kPtrHere : kPtrOther;
    return kPtrHost;
}

bool ctx_view(const void* ctx, CtxView* v) {
    const malib_ctx* c = static_cast<const malib_ctx*>(ctx);
    if (!c || !v) return false;
    v->device = c->device;
    v->stream = c->stream;
    v->n_sm = c->n_sm;
    v->has_pop = c->has_pop;
    v->env_kind = c->spec.env_kind;
    v->pol_dtype = c->pol_dtype;
    for (int i = 0; i < 4; ++i) v->dims[i] = c->dims[i];
    v->arena = c->arena;
    v->pol_offset = c->d_off;
    v->pol_seat = c->d_seat;
    v->n_pol = (int32_t)c->pols.size();
    v->err = c->d_err;
    v->tables_uploaded = !c->tables_dirty;
    v->tc_layout = c->tc_layout;
    return true;
}

int ctx_fail(void* ctx, int code, const char* msg) {
    return fail(static_cast<malib_ctx*>(ctx), code, "%s", msg);
}

int ctx_scratch(void* ctx, int64_t bytes, void** out) {
    malib_ctx* c = static_cast<malib_ctx*>(ctx);
    if (!c || !out || bytes < 0) return MALIB_EINVAL;
    DeviceGuard g(c->device);
    if (!g.ok) return fail(c, MALIB_ECUDA, "cannot select the context's device");
    const int r = ensure(c, c->scratch, c->scratch_cap, std::max<int64_t>(bytes, 1), "solver scratch");
    if (r != MALIB_OK) return r;
    *out = c->scratch;
    return MALIB_OK;
}

void ctx_count_launches(void* ctx, int n) {
    if (ctx) static_cast<malib_ctx*>(ctx)->launches += n;
}

}  // namespace malib

extern "C" {

int malib_create(malib_ctx** out, int device, void* cuda_stream) {
    if (!out) return fail(nullptr, MALIB_EINVAL, "out is NULL");
    *out = nullptr;
    int n_dev = 0;
    cudaError_t e = cudaGetDeviceCount(&n_dev);
    if (e != cudaSuccess || n_dev == 0)
        return fail(nullptr, MALIB_ECUDA, "no CUDA device: %s", cudaGetErrorString(e));
    if (device < 0 || device >= n_dev)
        return fail(nullptr, MALIB_EINVAL, "device %d out of range (%d devices)", device, n_dev);
    DeviceGuard g(device);
    malib_ctx* c = new malib_ctx();
    c->device = device;
    c->stream = (cudaStream_t)cuda_stream;
    cudaDeviceProp prop;
    if ((e = cudaGetDeviceProperties(&prop, device)) != cudaSuccess) {
        delete c;
        return fail(nullptr, MALIB_ECUDA, "device properties: %s", cudaGetErrorString(e));
    }
    c->n_sm = prop.multiProcessorCount;
    if ((e = cudaMalloc((void**)&c->d_err, 4)) != cudaSuccess ||
        (e = cudaMemset(c->d_err, 0, 4)) != cudaSuccess) {
        delete c;
        return fail(nullptr, MALIB_ENOMEM, "error flag: %s", cudaGetErrorString(e));
    }
    *out = c;
    return MALIB_OK;
}

void malib_destroy(malib_ctx* c) {
    if (!c) return;
    DeviceGuard g(c->device);
    cudaStreamSynchronize(c->stream);
    for (auto& ev : c->events) { cudaEventDestroy(ev.first); cudaEventDestroy(ev.second); }
    cudaFree(c->arena);
    cudaFree(c->d_off);
    cudaFree(c->d_seat);
    cudaFree(c->acc);
    cudaFree(c->d_err);
    cudaFree(c->d_pairs);
    cudaFree(c->d_out);
    cudaFree(c->scratch);
    cudaFree(c->lwork);
    cudaFree(c->learn_work);
    cudaFree(c->learn_grad);
    cudaFree(c->d_stage);
    cudaFree(c->d_jobs);
    delete c;
}

const char* malib_last_error(const malib_ctx* c) {
    return c ? c->err.c_str() : g_create_err.c_str();
}

int malib_sync(malib_ctx* c) {
    if (!c) return MALIB_EINVAL;
    DeviceGuard g(c->device);
    CK(cudaStreamSynchronize(c->stream), "stream");
    return read_device_errors(c);
}

int malib_set_stream(malib_ctx* c, void* s) {
    if (!c) return MALIB_EINVAL;
    c->stream = (cudaStream_t)s;
    return MALIB_OK;
}

int malib_pop_reset(malib_ctx* c) {
    if (!c) return MALIB_EINVAL;
    DeviceGuard g(c->device);
    CK(cudaStreamSynchronize(c->stream), "stream");
    c->pols.clear();
    c->arena_used = 0;
    c->has_pop = false;
    c->tables_dirty = true;
    return MALIB_OK;
}

int malib_pop_load(malib_ctx* c, const malib_env_spec* spec, const malib_policy_desc* pols,
                   int32_t n, int32_t* ids_out) {
    if (!c) return MALIB_EINVAL;
    DeviceGuard g(c->device);
    int r;
    if ((r = check_spec(c, spec)) != MALIB_OK) return r;
    if (n < 0 || (n > 0 && (!pols || !ids_out))) return fail(c, MALIB_EINVAL, "bad policy list");
    if (c->has_pop && !same_env(c->spec, *spec))
        return fail(c, MALIB_ESTATE, "population was loaded for a different environment");
    const bool poker = spec->env_kind == MALIB_ENV_KUHN || spec->env_kind == MALIB_ENV_LEDUC;
    std::vector<ConvJob> jobs(n);
    std::vector<PolicyRec> recs(n);
    int64_t stage_floats = 0, image_floats = 0, max_size = 0;
    for (int i = 0; i < n; ++i) {
        const malib_policy_desc& d = pols[i];
        PolicyRec rec{};
        rec.kind = d.kind;
        rec.dtype = d.dtype;
        rec.seat = d.seat;
        std::memcpy(rec.dims, d.dims, sizeof rec.dims);
        if (d.dtype != MALIB_F32 && d.dtype != MALIB_BF16)
            return fail(c, MALIB_EINVAL, "policy %d: unknown dtype %d", i, d.dtype);
        if (poker ? (d.seat < -1 || d.seat > 1) : false)
            return fail(c, MALIB_EINVAL, "policy %d: seat %d", i, d.seat);
        int64_t count;
        if (spec->env_kind == MALIB_ENV_KUHN) {
            if (d.kind != MALIB_POL_TABULAR || d.dims[0] != 6 || d.dims[3] != 1)
                return fail(c, MALIB_EINVAL, "policy %d: Kuhn needs a tabular policy of 6 infosets", i);
            count = 6;
        } else {
            if (d.kind != MALIB_POL_MLP || d.n_layers != 3)
                return fail(c, MALIB_EINVAL, "policy %d: needs a 3-layer MLP", i);
            if (d.dims[0] != spec->obs_dim || d.dims[3] != spec->n_actions || d.dims[1] < 1 ||
                d.dims[2] < 1)
                return fail(c, MALIB_EINVAL, "policy %d: dims %d-%d-%d-%d do not fit obs %d / actions %d",
                            i, d.dims[0], d.dims[1], d.dims[2], d.dims[3], spec->obs_dim,
                            spec->n_actions);
            count = mlp_param_floats(d.dims);
        }
        if (!d.params || d.nbytes != count * 4)
            return fail(c, MALIB_EINVAL, "policy %d: params NULL or nbytes %lld != %lld", i,
                        (long long)d.nbytes, (long long)(count * 4));
        const bool first = !c->has_pop && i == 0;
        const int* ref_dims = first ? d.dims : (c->has_pop ? c->dims : pols[0].dims);
        const int ref_kind = first ? d.kind : (c->has_pop ? c->pol_kind : pols[0].kind);
        const int ref_dtype = first ? d.dtype : (c->has_pop ? c->pol_dtype : pols[0].dtype);
        if (d.kind != ref_kind || d.dtype != ref_dtype || std::memcmp(d.dims, ref_dims, 16) != 0)
            return fail(c, MALIB_EINVAL, "policy %d: every policy of a population shares kind, dtype and dims", i);
        ConvJob& jb = jobs[i];
        conv_job(spec->env_kind, d.kind, d.dtype, d.dims, &jb);
        jb.src = stage_floats;
        jb.dst = c->arena_used + image_floats;
        rec.offset = jb.dst;
        stage_floats += (count + 3) / 4 * 4;            // 16-byte aligned sources
        image_floats += jb.size;
        max_size = std::max(max_size, jb.size);
        recs[i] = rec;
    }
    if (n > 0) {
        // the arena grows by a device copy of what it holds
        const int64_t need = c->arena_used + image_floats;
        if (need > c->arena_cap) {
            int64_t cap = c->arena_cap > 0 ? c->arena_cap : 1 << 16;
            while (cap < need) cap *= 2;
            float* na = nullptr;
            CK(cudaMalloc((void**)&na, (size_t)cap * 4), "population arena");
            if (c->arena_used > 0) {
                const cudaError_t e = cudaMemcpyAsync(na, c->arena, c->arena_used * 4,
                                                      cudaMemcpyDeviceToDevice, c->stream);
                if (e != cudaSuccess) {
                    cudaFree(na);
                    return cuda_fail(c, e, "arena copy");
                }
            }
            CK(cudaStreamSynchronize(c->stream), "arena copy");
            cudaFree(c->arena);
            c->arena = na;
            c->arena_cap = cap;
        }
        if ((r = ensure(c, c->d_stage, c->stage_cap, stage_floats, "parameter staging")) != MALIB_OK)
            return r;
        if ((r = ensure(c, c->d_jobs, c->jobs_cap, (int64_t)n, "conversion jobs")) != MALIB_OK)
            return r;
        // plain parameters from host or device memory (cudaMemcpyDefault: unified addressing)
        for (int i = 0; i < n; ++i)
            CK(cudaMemcpyAsync(c->d_stage + jobs[i].src, pols[i].params, pols[i].nbytes,
                               cudaMemcpyDefault, c->stream), "parameter upload");
        CK(cudaMemcpyAsync(c->d_jobs, jobs.data(), (size_t)n * sizeof(ConvJob), cudaMemcpyHostToDevice,
                           c->stream), "conversion jobs");
        for (int j0 = 0; j0 < n; j0 += 65535) {
            CK(launch_pop_convert(c->d_jobs + j0, std::min(65535, n - j0), max_size, c->d_stage,
                                  c->arena, c->stream), "population conversion kernel");
            c->launches += 1;
        }
        // the caller may free or reuse its parameter buffers once this returns
        CK(cudaStreamSynchronize(c->stream), "population load");
        c->arena_used = need;
    }
    for (int i = 0; i < n; ++i) {
        ids_out[i] = (int32_t)c->pols.size();
        c->pols.push_back(recs[i]);
    }
    if (!c->has_pop && n > 0) {
        c->has_pop = true;
        c->spec = *spec;
        c->pol_kind = pols[0].kind;
        c->pol_dtype = pols[0].dtype;
        std::memcpy(c->dims, pols[0].dims, sizeof c->dims);
        c->tc_layout = pols[0].kind == MALIB_POL_MLP && pols[0].dtype == MALIB_BF16 &&
                       tc_image_shape(pols[0].dims);
    }
    c->tables_dirty = true;
    if ((r = upload_tables(c)) != MALIB_OK) return r;
    return MALIB_OK;
}

int malib_eval_payoff_ex(malib_ctx* c, const int32_t* pair_ids, int32_t n_pairs,
                         int64_t n_episodes, uint64_t seed, uint32_t flags, double* payoff_out,
                         const malib_traj* dump, int64_t n_dump) {
    if (!c) return MALIB_EINVAL;
    DeviceGuard g(c->device);
    if (!c->has_pop) return fail(c, MALIB_ESTATE, "no population loaded");
    const int kind = c->spec.env_kind;
    if (kind != MALIB_ENV_KUHN && kind != MALIB_ENV_LEDUC)
        return fail(c, MALIB_ESTATE, "payoff evaluation needs a Kuhn or Leduc population");
    if (flags & ~(MALIB_DUMP_LOGITS | MALIB_EXACT_EXPECTATION))
        return fail(c, MALIB_EINVAL, "unknown flags 0x%x", flags);
    const bool exact = (flags & MALIB_EXACT_EXPECTATION) != 0;
    if (exact && kind != MALIB_ENV_KUHN)
        return fail(c, MALIB_EUNSUPPORTED, "exact expectation is built for Kuhn only");
    if (n_pairs < 0) return fail(c, MALIB_EINVAL, "n_pairs < 0");
    if (n_pairs == 0) return MALIB_OK;
    if (!pair_ids || !payoff_out) return fail(c, MALIB_EINVAL, "pair_ids or payoff_out is NULL");
    if (!exact && n_episodes < 1) return fail(c, MALIB_EINVAL, "n_episodes must be >= 1");
    if (!exact && n_episodes > ((int64_t)1 << 40) / n_pairs)
        return fail(c, MALIB_EINVAL, "n_pairs * n_episodes too large");
    if (kind == MALIB_ENV_KUHN && n_pairs > 65535)
        return fail(c, MALIB_EUNSUPPORTED, "Kuhn evaluation takes at most 65535 pairs per call");
    const bool want_dump = (flags & MALIB_DUMP_LOGITS) != 0 && !exact;
    if (want_dump) {
        if (!dump) return fail(c, MALIB_EINVAL, "MALIB_DUMP_LOGITS without a dump buffer");
        if (n_dump < 0 || n_dump > n_episodes) return fail(c, MALIB_EINVAL, "n_dump out of range");
        const void* ptrs[5] = {dump->obs, dump->action, dump->reward, dump->done, dump->logits};
        for (const void* p : ptrs)
            if (p && !is_device_ptr(c, p))
                return fail(c, MALIB_EINVAL, "dump buffers must be device memory of the context's device");
    }
    const bool leduc_tc = kind == MALIB_ENV_LEDUC && c->tc_layout && c->dims[0] == 17 &&
                          c->dims[3] == 3;
    if (kind == MALIB_ENV_LEDUC && !leduc_tc) {
        if (c->pol_dtype != MALIB_F32 || !leduc_f32_supported(c->dims[1]) || c->dims[1] != c->dims[2])
            return fail(c, MALIB_EUNSUPPORTED, "no Leduc kernel for %s hidden %d-%d",
                        c->pol_dtype == MALIB_BF16 ? "bf16" : "fp32", c->dims[1], c->dims[2]);
    }
    int r;
    if ((r = upload_tables(c)) != MALIB_OK) return r;
    const int32_t* dpairs = nullptr;
    if ((r = stage_pairs(c, pair_ids, (int64_t)n_pairs * 2, 2, true, &dpairs)) != MALIB_OK) return r;
    const int out_where = ptr_where(payoff_out, c->device);
    if (out_where == kPtrOther)
        return fail(c, MALIB_EINVAL, "payoff_out lives on another device than the context's");
    const bool host_out = out_where == kPtrHost;
    double* dout = payoff_out;
    if (host_out) {
        if ((r = ensure(c, c->d_out, c->out_cap, (int64_t)n_pairs * 4, "output staging")) != MALIB_OK)
            return r;
        dout = c->d_out;
    }
    EvalArgs a = eval_args(c);
    a.pairs = dpairs;
    a.n_pairs = n_pairs;
    a.n_episodes = n_episodes;
    a.seed = seed;
    if (want_dump) {
        a.n_dump = n_dump;
        a.d_obs = dump->obs;
        a.d_action = dump->action;
        a.d_reward = dump->reward;
        a.d_done = dump->done;
        a.d_logits = dump->logits;
    }
    cudaEvent_t e0, e1;
    if (exact) {
        time_begin(c, &e0, &e1);
        CK(launch_kuhn_exact(a, dout, c->stream), "Kuhn exact kernel");
        time_end(c, e0, e1);
        c->launches += 1;
    } else {
        // [n_pairs][2] sums, the decision count, [n_pairs] hand-claim counters
        if ((r = ensure(c, c->acc, c->acc_cap, (int64_t)n_pairs * 3 + 1, "payoff sums")) != MALIB_OK)
            return r;
        a.acc = c->acc;
        a.n_dec = c->acc + (int64_t)n_pairs * 2;
        a.work = c->acc + (int64_t)n_pairs * 2 + 1;
        c->last_pairs = n_pairs;
        CK(launch_zero_u64(c->acc, (int64_t)n_pairs * 3 + 1, c->stream), "zero kernel");
        time_begin(c, &e0, &e1);
        if (kind == MALIB_ENV_KUHN) {
            a.fin_out = dout;                 // each pair's last block writes its row
            CK(launch_kuhn_eval(a, c->n_sm, c->stream), "Kuhn eval kernel");
        } else if (leduc_tc) {
            int64_t n_seg = 0;
            int32_t split_from = 0;
            const int64_t units = leduc_tc_units(n_pairs, n_episodes, c->n_sm, &n_seg, &split_from);
            const int64_t grid = std::min<int64_t>(units, c->n_sm);
            const int64_t per = (n_episodes + n_seg - 1) / n_seg;
            LeducWork lw{};
            lw.max_hands = (int32_t)std::min<int64_t>(per, kLeducTcMaxHands);
            // per CTA: 8 bytes of state and 4 two-byte queue entries per hand
            if ((r = ensure(c, c->lwork, c->lwork_cap, grid * lw.max_hands * 16, "Leduc work space")) != MALIB_OK)
                return r;
            lw.hands = reinterpret_cast<uint2*>(c->lwork);
            lw.queues = reinterpret_cast<uint16_t*>(c->lwork + grid * lw.max_hands * 8);
            CK(launch_leduc_eval_tc(a, lw, c->n_sm, c->stream), "Leduc tensor-core eval kernel");
        } else {
            CK(launch_leduc_eval_f32(a, c->dims[1], c->n_sm, c->stream), "Leduc eval kernel");
        }
        time_end(c, e0, e1);
        if (!a.fin_out) CK(launch_finalize(c->acc, n_pairs, n_episodes, dout, c->stream), "finalize kernel");
        c->launches += a.fin_out ? 2 : 3;
    }
    if (host_out) {
        CK(cudaMemcpyAsync(payoff_out, dout, (size_t)n_pairs * 32, cudaMemcpyDeviceToHost,
                           c->stream), "payoff download");
        return read_device_errors(c);
    }
    return MALIB_OK;
}

int malib_eval_payoff(malib_ctx* c, const int32_t* pair_ids, int32_t n_pairs, int64_t n_episodes,
                      uint64_t seed, double* payoff_out) {
    return malib_eval_payoff_ex(c, pair_ids, n_pairs, n_episodes, seed, 0u, payoff_out, nullptr, 0);
}

int malib_rollout(malib_ctx* c, const malib_env_spec* spec, const int32_t* pair_ids,
                  int32_t n_pairs, int64_t n_episodes, uint64_t seed, malib_traj* traj) {
    if (!c) return MALIB_EINVAL;
    DeviceGuard g(c->device);
    int r;
    if ((r = check_spec(c, spec)) != MALIB_OK) return r;
    if (!c->has_pop) return fail(c, MALIB_ESTATE, "no population loaded");
    if (!same_env(c->spec, *spec))
        return fail(c, MALIB_ESTATE, "rollout spec differs from the population's environment");
    // scenarios of the fp32 rollout kernel other than spread (one policy width, hidden 64)
    const bool other = spec->env_kind == MALIB_ENV_ADVERSARY ||
                       spec->env_kind == MALIB_ENV_SPEAKER_LISTENER || spec->env_kind == MALIB_ENV_PUSH ||
                       spec->env_kind == MALIB_ENV_TAG || spec->env_kind == MALIB_ENV_REFERENCE;
    if (spec->env_kind != MALIB_ENV_SPREAD && !other)
        return fail(c, MALIB_EUNSUPPORTED, "rollout is built for the particle environments");
    if (n_pairs < 1) return fail(c, MALIB_EINVAL, "n_pairs must be >= 1");
    if (spec->n_envs < 1 || spec->n_envs % n_pairs != 0)
        return fail(c, MALIB_EINVAL, "n_envs (%lld) must be a positive multiple of n_pairs (%d)",
                    (long long)spec->n_envs, n_pairs);
    if (n_episodes < 0) return fail(c, MALIB_EINVAL, "n_episodes < 0");
    if (!pair_ids || !traj) return fail(c, MALIB_EINVAL, "pair_ids or traj_out is NULL");
    const bool want_logits = (spec->flags & MALIB_DUMP_LOGITS) != 0;
    if (!traj->obs || !traj->action || !traj->reward || !traj->done || (want_logits && !traj->logits))
        return fail(c, MALIB_EINVAL, "trajectory buffer missing");
    const void* ptrs[5] = {traj->obs, traj->action, traj->reward, traj->done,
                           want_logits ? traj->logits : traj->obs};
    for (const void* p : ptrs) {
        if (!is_device_ptr(c, p))
            return fail(c, MALIB_EINVAL, "trajectory buffers must be device memory of the context's device");
        if (((uintptr_t)p & 15u) != 0) return fail(c, MALIB_EINVAL, "trajectory buffers must be 16-byte aligned");
    }
    const int64_t epp = spec->n_envs / n_pairs;
    const bool use_tc = !other && c->tc_layout && spread_tc_supported(spec->n_agents, spec->obs_dim,
                                                                    spec->n_actions, epp);
    const bool f32_ok = other ? scenario_f32_supported(c->dims[1])
                            : spread_f32_supported(spec->n_agents, spec->obs_dim, c->dims[1]);
    if (!use_tc && (c->pol_dtype != MALIB_F32 || c->dims[1] != c->dims[2] || !f32_ok || epp > 128))
        return fail(c, MALIB_EUNSUPPORTED,
                    "no spread kernel for %s N=%d obs %d hidden %d with %lld envs per combination",
                    c->pol_dtype == MALIB_BF16 ? "bf16" : "fp32", spec->n_agents, spec->obs_dim,
                    c->dims[1], (long long)epp);
    if (n_episodes == 0) return MALIB_OK;
    if ((r = upload_tables(c)) != MALIB_OK) return r;
    const int32_t* dpairs = nullptr;
    if ((r = stage_pairs(c, pair_ids, (int64_t)n_pairs * spec->n_agents, spec->n_agents, false,
                         &dpairs)) != MALIB_OK)
        return r;
    RolloutArgs a{};
    a.env_kind = spec->env_kind;
    a.arena = c->arena;
    a.pol_offset = c->d_off;
    a.n_pol = (int32_t)c->pols.size();
    a.pairs = dpairs;
    a.n_pairs = n_pairs;
    a.n_agents = spec->n_agents;
    a.obs_dim = spec->obs_dim;
    a.obs_pad = (spec->obs_dim + 3) / 4 * 4;
    a.episode_len = spec->episode_len;
    a.local_ratio = (spec->flags & MALIB_SPREAD_LOCAL_RATIO) ? spec->local_ratio : -1.0f;
    a.contact = (spec->flags & MALIB_SPREAD_CONTACT) ? 1 : 0;
    a.n_envs = spec->n_envs;
    a.n_episodes = n_episodes;
    a.seed = seed;
    a.err = c->d_err;
    a.obs = traj->obs;
    a.action = traj->action;
    a.reward = traj->reward;
    a.done = traj->done;
    a.logits = want_logits ? traj->logits : nullptr;
    cudaEvent_t e0, e1;
    time_begin(c, &e0, &e1);
    if (use_tc) {
        CK(launch_spread_rollout_tc(a, c->n_sm, c->stream), "spread tensor-core rollout kernel");
    } else {
        CK(launch_spread_rollout_f32(a, c->dims[1], c->n_sm, c->stream), "spread rollout kernel");
    }
    time_end(c, e0, e1);
    c->launches += 1;
    return MALIB_OK;
}

namespace {

// The policy-gradient step of nb distinct policies (host ids) in one batch.
// clip > 0: the PPO surrogate against the behavior logits traj->logits; 0: the policy gradient.
int learn_batch(malib_ctx* c, const malib_env_spec* spec, const int32_t* pair_ids, int32_t n_pairs,
                int64_t n_episodes, const malib_traj* traj, const int32_t* ids, int32_t nb, float gamma,
                float entropy_coef, float clip, float* grad_out, double* stats_out) {
    int r;
    if ((r = check_spec(c, spec)) != MALIB_OK) return r;
    if (!c->has_pop) return fail(c, MALIB_ESTATE, "no population loaded");
    if (!same_env(c->spec, *spec))
        return fail(c, MALIB_ESTATE, "spec differs from the population's environment");
    if (spec->env_kind == MALIB_ENV_KUHN || spec->env_kind == MALIB_ENV_LEDUC)
        return fail(c, MALIB_EUNSUPPORTED, "the learner step is built for the particle rollouts");
    if (c->pol_kind != MALIB_POL_MLP || c->pol_dtype != MALIB_F32 ||
        !learn_supported(c->dims[0], c->dims[1], c->dims[2], c->dims[3]))
        return fail(c, MALIB_EUNSUPPORTED, "the learner step is built for fp32 MLPs in-64-64-5 (in <= %d)",
                    kLearnMaxIn);
    if (nb < 1 || !ids) return fail(c, MALIB_EINVAL, "the batch needs at least one policy id");
    std::vector<int32_t> hid(ids, ids + nb);
    std::vector<int64_t> hoff(nb);
    for (int32_t b = 0; b < nb; ++b) {
        if (hid[b] < 0 || hid[b] >= (int32_t)c->pols.size())
            return fail(c, MALIB_EINVAL, "policy id %d is not in the population", hid[b]);
        for (int32_t q = 0; q < b; ++q)
            if (hid[q] == hid[b]) return fail(c, MALIB_EINVAL, "policy id %d appears twice in the batch", hid[b]);
        hoff[b] = c->pols[hid[b]].offset;
    }
    if (n_pairs < 1) return fail(c, MALIB_EINVAL, "n_pairs must be >= 1");
    if (spec->n_envs < 1 || spec->n_envs % n_pairs != 0)
        return fail(c, MALIB_EINVAL, "n_envs (%lld) must be a positive multiple of n_pairs (%d)",
                    (long long)spec->n_envs, n_pairs);
    if (n_episodes < 0) return fail(c, MALIB_EINVAL, "n_episodes < 0");
    if (!(gamma >= 0.0f && gamma <= 1.0f)) return fail(c, MALIB_EINVAL, "gamma must lie in [0, 1]");
    if (!(entropy_coef >= 0.0f && entropy_coef < 1e30f)) return fail(c, MALIB_EINVAL, "entropy_coef must be >= 0");
    if (!pair_ids || !traj || !grad_out) return fail(c, MALIB_EINVAL, "pair_ids, traj or grad_out is NULL");
    if (!traj->obs || !traj->action || !traj->reward) return fail(c, MALIB_EINVAL, "trajectory buffer missing");
    const void* tp[3] = {traj->obs, traj->action, traj->reward};
    for (const void* p : tp)
        if (!is_device_ptr(c, p))
            return fail(c, MALIB_EINVAL, "trajectory buffers must be device memory of the context's device");
    if (clip != 0.0f) {
        if (!(clip > 0.0f && clip < 1.0f)) return fail(c, MALIB_EINVAL, "clip_eps must lie in (0, 1)");
        if (!traj->logits || !is_device_ptr(c, traj->logits))
            return fail(c, MALIB_EINVAL, "the PPO step needs the behavior logits (traj->logits, device memory)");
    }
    const int gw = ptr_where(grad_out, c->device);
    const int sw = stats_out ? ptr_where(stats_out, c->device) : kPtrHost;
    if (gw == kPtrOther || sw == kPtrOther)
        return fail(c, MALIB_EINVAL, "grad_out or stats_out lives on another device than the context's");
    if ((r = upload_tables(c)) != MALIB_OK) return r;
    const int32_t* dpairs = nullptr;
    if ((r = stage_pairs(c, pair_ids, (int64_t)n_pairs * spec->n_agents, spec->n_agents, false, &dpairs)) !=
        MALIB_OK)
        return r;
    const int in = c->dims[0];
    const int64_t P = learn_param_count(in);
    const int grid = c->n_sm;
    const int ret_blocks = 2 * c->n_sm;
    const int64_t bytes = learn_work_bytes(nb, n_pairs, spec->n_agents, spec->n_envs, n_episodes,
                                           spec->episode_len, in, grid, ret_blocks);
    if ((r = ensure(c, c->learn_work, c->learn_work_cap, bytes, "learner work space")) != MALIB_OK) return r;
    LearnArgs a{};
    learn_work_layout(c->learn_work, nb, n_pairs, spec->n_agents, spec->n_envs, n_episodes, spec->episode_len, in,
                      grid, ret_blocks, &a);
    if (gw == kPtrHere) {
        a.grad = grad_out;
    } else {
        if ((r = ensure(c, c->learn_grad, c->learn_grad_cap, (int64_t)nb * P, "gradient staging")) != MALIB_OK)
            return r;
        a.grad = c->learn_grad;
    }
    CK(cudaMemcpyAsync(const_cast<int32_t*>(a.pols), hid.data(), (size_t)nb * 4, cudaMemcpyHostToDevice,
                       c->stream), "policy ids");
    CK(cudaMemcpyAsync(const_cast<int64_t*>(a.pol_offs), hoff.data(), (size_t)nb * 8, cudaMemcpyHostToDevice,
                       c->stream), "policy offsets");
    a.arena = c->arena;
    a.in = in;
    a.xs = (spec->obs_dim + 3) / 4 * 4;
    a.pairs = dpairs;
    a.n_pairs = n_pairs;
    a.n_agents = spec->n_agents;
    a.n_pol = (int32_t)c->pols.size();
    a.T = spec->episode_len;
    a.n_envs = spec->n_envs;
    a.n_episodes = n_episodes;
    a.obs = traj->obs;
    a.action = traj->action;
    a.reward = traj->reward;
    a.gamma = gamma;
    a.beta = entropy_coef;
    a.clip = clip;
    a.blogits = clip > 0.0f ? traj->logits : nullptr;
    a.err = c->d_err;
    // with timing on, the gradient kernel (the step's dominant one) is the timed launch
    cudaEvent_t g0 = nullptr, g1 = nullptr;
    if (c->timing && (cudaEventCreate(&g0) != cudaSuccess || cudaEventCreate(&g1) != cudaSuccess)) {
        cudaGetLastError();
        if (g0) cudaEventDestroy(g0);
        g0 = g1 = nullptr;
    }
    CK(launch_learn_pg(a, ret_blocks, c->stream, g0, g1), "policy-gradient kernels");
    if (g0) c->events.emplace_back(g0, g1);
    c->launches += 6;
    if (gw != kPtrHere)
        CK(cudaMemcpyAsync(grad_out, a.grad, (size_t)nb * P * 4, cudaMemcpyDeviceToHost, c->stream),
           "gradient copy");
    if (stats_out)
        CK(cudaMemcpyAsync(stats_out, a.stats, (size_t)nb * 4 * 8,
                           sw == kPtrHere ? cudaMemcpyDeviceToDevice : cudaMemcpyDeviceToHost, c->stream),
           "statistics copy");
    // the host vectors of ids and offsets are copied before they go out of scope
    CK(cudaStreamSynchronize(c->stream), "learner step");
    return read_device_errors(c);
}

}  // namespace

int malib_learn_pg(malib_ctx* c, const malib_env_spec* spec, const int32_t* pair_ids, int32_t n_pairs,
                   int64_t n_episodes, const malib_traj* traj, int32_t policy_id, float gamma,
                   float entropy_coef, float* grad_out, double* stats_out) {
    if (!c) return MALIB_EINVAL;
    DeviceGuard g(c->device);
    return learn_batch(c, spec, pair_ids, n_pairs, n_episodes, traj, &policy_id, 1, gamma, entropy_coef, 0.0f,
                       grad_out, stats_out);
}

int malib_learn_pg_batch(malib_ctx* c, const malib_env_spec* spec, const int32_t* pair_ids, int32_t n_pairs,
                         int64_t n_episodes, const malib_traj* traj, const int32_t* policy_ids,
                         int32_t n_policies, float gamma, float entropy_coef, float* grad_out, double* stats_out) {
    if (!c) return MALIB_EINVAL;
    DeviceGuard g(c->device);
    return learn_batch(c, spec, pair_ids, n_pairs, n_episodes, traj, policy_ids, n_policies, gamma, entropy_coef,
                       0.0f, grad_out, stats_out);
}

int malib_learn_ppo_batch(malib_ctx* c, const malib_env_spec* spec, const int32_t* pair_ids, int32_t n_pairs,
                          int64_t n_episodes, const malib_traj* traj, const int32_t* policy_ids,
                          int32_t n_policies, float gamma, float entropy_coef, float clip_eps, float* grad_out,
                          double* stats_out) {
    if (!c) return MALIB_EINVAL;
    DeviceGuard g(c->device);
    if (!(clip_eps > 0.0f && clip_eps < 1.0f)) return fail(c, MALIB_EINVAL, "clip_eps must lie in (0, 1)");
    return learn_batch(c, spec, pair_ids, n_pairs, n_episodes, traj, policy_ids, n_policies, gamma, entropy_coef,
                       clip_eps, grad_out, stats_out);
}

int malib_adam_step(malib_ctx* c, float* params, const float* grad, float* m, float* v, int64_t n, int64_t step,
                    float lr, float beta1, float beta2, float eps) {
    if (!c) return MALIB_EINVAL;
    DeviceGuard g(c->device);
    if (n < 0) return fail(c, MALIB_EINVAL, "n < 0");
    if (n == 0) return MALIB_OK;
    if (!params || !grad || !m || !v) return fail(c, MALIB_EINVAL, "a buffer is NULL");
    const void* ptrs[4] = {params, grad, m, v};
    for (const void* p : ptrs)
        if (!is_device_ptr(c, p)) return fail(c, MALIB_EINVAL, "Adam buffers must be device memory of the context's device");
    if (step < 1) return fail(c, MALIB_EINVAL, "step must be >= 1");
    if (!(lr >= 0.0f) || !(beta1 >= 0.0f && beta1 < 1.0f) || !(beta2 >= 0.0f && beta2 < 1.0f) || !(eps > 0.0f))
        return fail(c, MALIB_EINVAL, "need lr >= 0, 0 <= beta1, beta2 < 1, eps > 0");
    const float c1 = (float)(1.0 - std::pow((double)beta1, (double)step));
    const float c2 = (float)(1.0 - std::pow((double)beta2, (double)step));
    CK(launch_learn_adam(params, grad, m, v, n, lr, beta1, beta2, eps, c1 > 0.f ? c1 : 1.f, c2 > 0.f ? c2 : 1.f,
                         c->n_sm, c->stream),
       "Adam kernel");
    c->launches += 1;
    return MALIB_OK;
}

int malib_pop_update(malib_ctx* c, int32_t policy_id, const float* params, int64_t nbytes) {
    if (!c) return MALIB_EINVAL;
    DeviceGuard g(c->device);
    if (!c->has_pop) return fail(c, MALIB_ESTATE, "no population loaded");
    if (policy_id < 0 || policy_id >= (int32_t)c->pols.size())
        return fail(c, MALIB_EINVAL, "policy_id %d is not in the population", policy_id);
    const PolicyRec& rec = c->pols[policy_id];
    const int64_t count = rec.kind == MALIB_POL_TABULAR ? 6 : mlp_param_floats(rec.dims);
    if (!params || nbytes != count * 4)
        return fail(c, MALIB_EINVAL, "params NULL or nbytes %lld != %lld", (long long)nbytes,
                    (long long)(count * 4));
    if (ptr_where(params, c->device) == kPtrOther)
        return fail(c, MALIB_EINVAL, "params live on another device than the context's");
    ConvJob jb{};
    conv_job(c->spec.env_kind, rec.kind, rec.dtype, rec.dims, &jb);
    jb.src = 0;
    jb.dst = rec.offset;
    int r;
    if ((r = ensure(c, c->d_stage, c->stage_cap, (count + 3) / 4 * 4, "parameter staging")) != MALIB_OK) return r;
    if ((r = ensure(c, c->d_jobs, c->jobs_cap, (int64_t)1, "conversion jobs")) != MALIB_OK) return r;
    CK(cudaMemcpyAsync(c->d_stage, params, nbytes, cudaMemcpyDefault, c->stream), "parameter upload");
    CK(cudaMemcpyAsync(c->d_jobs, &jb, sizeof jb, cudaMemcpyHostToDevice, c->stream), "conversion job");
    CK(launch_pop_convert(c->d_jobs, 1, jb.size, c->d_stage, c->arena, c->stream), "population conversion kernel");
    c->launches += 1;
    // the caller may free or reuse its buffer once this returns
    CK(cudaStreamSynchronize(c->stream), "population update");
    return MALIB_OK;
}

int malib_eval_stats(malib_ctx* c, int64_t* n_decisions) {
    if (!c || !n_decisions) return MALIB_EINVAL;
    DeviceGuard g(c->device);
    *n_decisions = 0;
    if (c->last_pairs < 0) return fail(c, MALIB_ESTATE, "no Monte-Carlo evaluation has run");
    unsigned long long v = 0;
    CK(cudaMemcpyAsync(&v, c->acc + c->last_pairs * 2, 8, cudaMemcpyDeviceToHost, c->stream),
       "decision count");
    CK(cudaStreamSynchronize(c->stream), "sync");
    *n_decisions = (int64_t)v;
    return MALIB_OK;
}

int64_t malib_launch_count(const malib_ctx* c) { return c ? c->launches : 0; }

int malib_set_timing(malib_ctx* c, int enable) {
    if (!c) return MALIB_EINVAL;
    c->timing = enable != 0;
    return MALIB_OK;
}

double malib_main_kernel_ms(malib_ctx* c, int64_t* n_launches, int reset) {
    if (!c) return -1.0;
    DeviceGuard g(c->device);
    for (auto& ev : c->events) {
        float ms = 0.f;
        if (cudaEventSynchronize(ev.second) == cudaSuccess &&
            cudaEventElapsedTime(&ms, ev.first, ev.second) == cudaSuccess) {
            c->timed_ms += ms;
            c->timed_n += 1;
        }
        cudaGetLastError();
        cudaEventDestroy(ev.first);
        cudaEventDestroy(ev.second);
    }
    c->events.clear();
    const double ms = c->timed_ms;
    if (n_launches) *n_launches = c->timed_n;
    if (reset) { c->timed_ms = 0.0; c->timed_n = 0; }
    return ms;
}

int malib_selftest_philox(malib_ctx* c, const uint32_t* ctr, uint64_t seed, uint32_t* out,
                          int64_t n) {
    if (!c) return MALIB_EINVAL;
    DeviceGuard g(c->device);
    if (n < 0 || (n > 0 && (!ctr || !out || !is_device_ptr(c, ctr) || !is_device_ptr(c, out))))
        return fail(c, MALIB_EINVAL, "philox self-test needs device buffers");
    CK(launch_selftest_philox(ctr, seed, out, n, c->stream), "philox kernel");
    c->launches += n > 0;
    return MALIB_OK;
}

int malib_philox_digest(malib_ctx* c, uint64_t seed, int64_t n, int32_t calls, uint32_t* out) {
    if (!c) return MALIB_EINVAL;
    DeviceGuard g(c->device);
    if (n < 0 || calls < 0 || (n > 0 && (!out || !is_device_ptr(c, out))))
        return fail(c, MALIB_EINVAL, "philox digest needs n >= 0, calls >= 0 and a device buffer");
    CK(launch_philox_digest(seed, n, calls, out, c->stream), "philox digest kernel");
    c->launches += n > 0;
    return MALIB_OK;
}

int malib_selftest_wait(malib_ctx* c, int32_t arrive, int64_t limit_ns) {
    if (!c) return MALIB_EINVAL;
    DeviceGuard g(c->device);
    if (limit_ns < 1 || limit_ns > 1000000000)
        return fail(c, MALIB_EINVAL, "limit_ns must lie in [1, 1e9]");
    CK(launch_selftest_wait(arrive != 0, (uint64_t)limit_ns, c->d_err, c->stream), "wait self-test kernel");
    c->launches += 1;
    return MALIB_OK;
}

int malib_selftest_det_expf(malib_ctx* c, const float* x, float* y, int64_t n) {
    if (!c) return MALIB_EINVAL;
    DeviceGuard g(c->device);
    if (n < 0 || (n > 0 && (!x || !y || !is_device_ptr(c, x) || !is_device_ptr(c, y))))
        return fail(c, MALIB_EINVAL, "det_expf self-test needs device buffers");
    CK(launch_selftest_det_expf(x, y, n, c->stream), "det_expf kernel");
    c->launches += n > 0;
    return MALIB_OK;
}

int malib_selftest_sample(malib_ctx* c, const float* logits, const uint8_t* legal, const float* u,
                          int32_t A, int32_t* out, int64_t n) {
    if (!c) return MALIB_EINVAL;
    DeviceGuard g(c->device);
    if (A < 2 || A > 8) return fail(c, MALIB_EINVAL, "A must be in [2, 8]");
    if (n < 0 || (n > 0 && (!logits || !legal || !u || !out || !is_device_ptr(c, logits) ||
                            !is_device_ptr(c, legal) || !is_device_ptr(c, u) || !is_device_ptr(c, out))))
        return fail(c, MALIB_EINVAL, "sample self-test needs device buffers");
    CK(launch_selftest_sample(logits, legal, u, A, out, n, c->stream), "sample kernel");
    c->launches += n > 0;
    return MALIB_OK;
}

}  // extern "C"
