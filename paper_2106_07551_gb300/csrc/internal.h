// Internal interface between the host runtime (runtime.cu) and the kernels.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "malib.h"

namespace malib {

constexpr int kMaxAgents = 16;

// Error bits raised by kernels into the context's device error word.
enum : int {
    ERRBIT_BAD_PAIR = 1,      // an id in a device pair table is out of range / wrong seat
    ERRBIT_TIMEOUT = 2,       // a bounded mbarrier wait expired
    ERRBIT_NOT_CONVERGED = 4, // an iterative solver reached its iteration limit
};

// fp32 MLP policy, kernel layout of one population member (floats, every
// sub-array 16-byte aligned):
//   W1T[IN][H]   (k-major: W1T[k][j] = W1[j][k])
//   b1[H]
//   W2T[H][H]    (k-major)
//   b2[H]
//   W3[A][H]     (row-major as given)
//   b3[A], padded to a multiple of 4
template <int IN, int H, int A>
struct F32Layout {
    static constexpr int kW1T = 0;
    static constexpr int kB1 = IN * H;
    static constexpr int kW2T = kB1 + H;
    static constexpr int kB2 = kW2T + H * H;
    static constexpr int kW3 = kB2 + H;
    static constexpr int kB3 = kW3 + A * H;
    static constexpr int kSize = (kB3 + A + 3) / 4 * 4;
    static_assert(IN * H % 4 == 0 && H % 8 == 0, "layout alignment");
};

// bf16 tensor-core policy image (bytes): W1 [256][K1], W2 [256][256], W3 [16][256]
// as bf16 in the core-matrix K-major layout (K1 = input width rounded up to
// 16, rows past the output width zero), then fp32 b1[256], b2[256], b3[16].
// Built for populations with h1 = h2 = 256, input <= 48, output <= 16.
inline bool tc_image_shape(const int* d) {
    return d[1] == 256 && d[2] == 256 && d[0] >= 1 && d[0] <= 48 && d[3] >= 1 && d[3] <= 16;
}
// Leduc's observation feature 15 (call/check legal) is 1 in every state: the
// Leduc tensor-core image folds its weight column into b1 and drops the
// feature, leaving 16 inputs (one bf16 K step).
constexpr int kLeducConstFeature = 15;
inline bool leduc_tc_fold(int env_kind, int in) { return env_kind == MALIB_ENV_LEDUC && in == 17; }
inline int64_t tc_image_bytes(int in) {
    const int64_t k1 = (in + 15) / 16 * 16;
    return 256 * k1 * 2 + 256 * 256 * 2 + 16 * 256 * 2 + (256 + 256 + 16) * 4;
}

// Output sums of the payoff reduction: per pair {sum r, sum r^2} as 64-bit
// two's complement (integers, so any summation order gives the same bits).
struct EvalArgs {
    const float* arena;          // population arena (kernel layouts)
    const int64_t* pol_offset;   // [n_pol] float offset of each policy in arena
    const int32_t* pol_seat;     // [n_pol] owning seat (-1 shared)
    int32_t n_pol;
    const int32_t* pairs;        // device [n_pairs][2]
    int32_t n_pairs;
    int64_t n_episodes;
    uint64_t seed;
    unsigned long long* acc;     // [n_pairs][2]
    unsigned long long* n_dec;   // total decisions (env-steps) of the call
    unsigned long long* work;    // [n_pairs] hands claimed so far (zeroed per call)
    double* fin_out;             // Kuhn: [n_pairs][4] table written by each pair's last
                                 // block (work[] counts its finished blocks); null: a
                                 // separate finalize launch writes it
    int* err;
    // optional dump of the first n_dump episodes of each pair
    int64_t n_dump;
    float* d_obs;
    uint8_t* d_action;
    float* d_reward;
    uint8_t* d_done;
    float* d_logits;
};

struct RolloutArgs {
    int32_t env_kind;            // MALIB_ENV_SPREAD or another particle scenario
    const float* arena;
    const int64_t* pol_offset;
    int32_t n_pol;
    const int32_t* pairs;        // device [n_pairs][N]
    int32_t n_pairs;
    int32_t n_agents;
    int32_t obs_dim;
    int32_t obs_pad;             // obs_dim rounded up to 4
    int32_t episode_len;
    int64_t n_envs;
    int64_t n_episodes;
    uint64_t seed;
    int* err;
    float* obs;
    uint8_t* action;
    float* reward;
    uint8_t* done;
    float* logits;               // may be null
    float local_ratio;           // < 0: r_i = -(cover + coll_i); else the weighted reward
    int32_t contact;             // SPREAD: agents push each other apart (soft contact forces)
};

// Launchers (return cudaGetLastError() of the launch). `grid_hint` = SM count.
cudaError_t launch_kuhn_eval(const EvalArgs& a, int n_sm, cudaStream_t s);
cudaError_t launch_kuhn_exact(const EvalArgs& a, double* out, cudaStream_t s);
cudaError_t launch_leduc_eval_f32(const EvalArgs& a, int hidden, int n_sm, cudaStream_t s);
// Work space of the tensor-core Leduc evaluation: per CTA, the state of up to
// max_hands hands (two words each) and four queues of hand slots.
constexpr int kLeducTcMaxHands = 16384;
struct LeducWork {
    uint2* hands;                // [grid][max_hands]
    uint16_t* queues;            // [grid][2 seats][2 queues][max_hands]
    int32_t max_hands;
    int64_t n_seg;               // segments per pair (set by the launcher)
    int32_t split_from;          // pairs from this one on are played in 2 n_seg segments
    int64_t n_units;             // units of the call
};
// Units (pair, segment) of a call: n_seg segments per pair, and twice as many
// for the pairs from *split_from on (the last ones claimed, so that the CTAs
// finish closer together).
int64_t leduc_tc_units(int32_t n_pairs, int64_t n_episodes, int n_sm, int64_t* n_seg_out,
                       int32_t* split_from_out);
cudaError_t launch_leduc_eval_tc(const EvalArgs& a, const LeducWork& w, int n_sm, cudaStream_t s);
cudaError_t launch_spread_rollout_f32(const RolloutArgs& a, int hidden, int n_sm, cudaStream_t s);
cudaError_t launch_spread_rollout_tc(const RolloutArgs& a, int n_sm, cudaStream_t s);
bool spread_tc_supported(int n_agents, int obs_dim, int n_actions, int64_t envs_per_pair);
// Learner-side policy-gradient step (learner.cu) on a rollout's samples of a
// batch of policies (each its own independent learner): fp32 MLPs in-64-64-5
// with in <= kLearnMaxIn.
constexpr int kLearnMaxIn = 32;
struct LearnArgs {
    const float* arena;          // population arena (F32Layout images)
    const int32_t* pols;         // device [nb] policy ids of the batch (distinct)
    const int64_t* pol_offs;     // device [nb] float offsets of their images
    int32_t nb;                  // policies in the batch
    int32_t in;                  // observation width (policy input)
    int32_t xs;                  // observation row stride of the trajectory (in rounded up to 4)
    const int32_t* pairs;        // device [n_pairs][n_agents]
    int32_t n_pairs, n_agents, n_pol, T;
    int64_t n_envs, n_episodes;
    const float* obs;            // [E][T][n_envs][n_agents][xs]
    const uint8_t* action;       // [E][T][n_envs][n_agents]
    const float* reward;         // [E][T][n_envs][n_agents]
    float gamma, beta;
    // PPO (clip > 0): the behavior policy's logits [E][T][n_envs][n_agents][5]
    // that the rollout recorded, and the clip range; clip == 0: the policy gradient
    const float* blogits;
    float clip;
    int* err;
    // work space (learn_work_layout)
    int32_t* slots;              // [nb][n_pairs * n_agents] (c * n_agents + k) acting with each policy
    int32_t* n_slots;            // [nb]
    int64_t* samp_off;           // [nb + 1] first sample of each policy in G
    int64_t* tile_off;           // [nb + 1] first 128-sample tile of each policy
    float* G;                    // [samples] returns-to-go, policy by policy in sample order
    double* gsum;                // [nb][return blocks] partial sums of G
    double* stats;               // [nb][4] M, baseline, loss, mean entropy
    float* gpart;                // [nb][grid][P + 2] per-CTA partial gradients, loss and entropy sums
    float* grad;                 // [nb][P] the gradients (malib_policy_desc layout)
    int32_t grid;
};
int64_t learn_param_count(int in);
bool learn_supported(int in, int h1, int h2, int n_actions);
int64_t learn_work_bytes(int32_t nb, int32_t n_pairs, int32_t n_agents, int64_t n_envs, int64_t n_episodes,
                         int32_t T, int in, int grid, int ret_blocks);
void learn_work_layout(uint8_t* base, int32_t nb, int32_t n_pairs, int32_t n_agents, int64_t n_envs,
                       int64_t n_episodes, int32_t T, int in, int grid, int ret_blocks, LearnArgs* a);
// g0 / g1 (optional): events recorded just before and after learn_grad_kernel.
cudaError_t launch_learn_pg(const LearnArgs& a, int ret_blocks, cudaStream_t s, cudaEvent_t g0 = nullptr,
                            cudaEvent_t g1 = nullptr);
cudaError_t launch_learn_adam(float* p, const float* g, float* m, float* v, int64_t n, float lr, float b1,
                              float b2, float eps, float c1, float c2, int n_sm, cudaStream_t s);
cudaError_t launch_zero_u64(unsigned long long* p, int64_t n, cudaStream_t s);
cudaError_t launch_finalize(const unsigned long long* acc, int32_t n_pairs, int64_t n_episodes,
                            double* out, cudaStream_t s);
cudaError_t launch_selftest_wait(bool arrive, uint64_t limit_ns, int* err, cudaStream_t s);
// One policy of a population load: its plain fp32 parameters at stage + src
// (row-major W[out][in] then b[out], per layer) become its kernel image at
// arena + dst, `size` 32-bit words (pop_convert.cu).
constexpr int32_t kConvTable = 0, kConvF32 = 1, kConvTc = 2;   // kind
constexpr int32_t kConvRound = 1, kConvFold = 2;               // flags
struct ConvJob {
    int64_t src;        // float offset in the staging buffer
    int64_t dst;        // float offset in the arena
    int64_t size;       // image words
    int32_t kind;
    int32_t flags;      // kConvRound: weights to bf16 (fp32 layout); kConvFold: Leduc feature 15
    int32_t dims[4];
};
cudaError_t launch_pop_convert(const ConvJob* jobs, int n_jobs, int64_t max_size, const float* stage,
                               float* arena, cudaStream_t s);

cudaError_t launch_philox_digest(uint64_t seed, int64_t n, int calls, uint32_t* out,
                                 cudaStream_t s);
cudaError_t launch_selftest_philox(const uint32_t* ctr, uint64_t seed, uint32_t* out, int64_t n,
                                   cudaStream_t s);
cudaError_t launch_selftest_det_expf(const float* x, float* y, int64_t n, cudaStream_t s);
cudaError_t launch_selftest_sample(const float* logits, const uint8_t* legal, const float* u,
                                   int A, int32_t* out, int64_t n, cudaStream_t s);

// Read-only view of a context for entry points defined outside runtime.cu.
struct CtxView {
    int device;
    cudaStream_t stream;
    int n_sm;
    bool has_pop;
    int env_kind;
    int pol_dtype;
    int dims[4];
    const float* arena;
    const int64_t* pol_offset;
    const int32_t* pol_seat;
    int32_t n_pol;
    int* err;
    bool tables_uploaded;
    bool tc_layout;               // bf16 tensor-core images in the arena (else fp32 layouts)
};
bool ctx_view(const void* ctx, CtxView* v);
// Where a pointer lives, by cudaPointerGetAttributes: host memory (pageable,
// pinned or unknown), device memory of `device` (or managed memory), or device
// memory of another GPU, which no kernel of a context on `device` may touch.
enum : int { kPtrHost = 0, kPtrHere = 1, kPtrOther = -1 };
int ptr_where(const void* p, int device);
int ctx_fail(void* ctx, int code, const char* msg);
void ctx_count_launches(void* ctx, int n);
// Device work space owned by the context, grown on its stream (cudaMallocAsync).
int ctx_scratch(void* ctx, int64_t bytes, void** out);

// Meta-game solvers (meta_solver.cu).
cudaError_t launch_fictitious_play(const double* P, int32_t G, int32_t m, int32_t n, int32_t stride,
                                   int64_t T, double* x, double* y, double* bounds, int n_sm,
                                   cudaStream_t s);
cudaError_t launch_aggregate(const double* P, int32_t G, int32_t m, int32_t n, int32_t stride,
                             const double* x, const double* y, double* ay, double* xa, double* val,
                             int n_sm, cudaStream_t s);
int64_t lp_tableau_doubles(int32_t m, int32_t n);
bool lp_on_chip(int32_t m, int32_t n);
int lp_grid(int32_t n_games, int n_sm);
cudaError_t launch_lp_nash(const double* P, int32_t G, int32_t m, int32_t n, int32_t stride,
                           double* x, double* y, double* val, double* scratch, int32_t pivot_limit,
                           int* err, int n_sm, cudaStream_t s);

bool leduc_f32_supported(int hidden);
bool spread_f32_supported(int n_agents, int obs_dim, int hidden);
// The simple adversary and simple speaker listener scenarios (hidden width 64).
bool scenario_f32_supported(int hidden);

}  // namespace malib
