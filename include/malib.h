/*
 * malib.h - C ABI of the GB300 rollout and payoff-evaluation path of MALib
 * (Zhou et al., "MALib: A Parallel Framework for Population-based Multi-agent
 * Reinforcement Learning", arXiv 2106.07551).
 *
 * Vocabulary (Sec. 3.1 "Defining the Task Graph"): a *population* holds policy
 * pools; a *policy combination* Comb_t picks one policy per agent; a *rollout*
 * draws trajectories X ~ P(s, a, s' | a ~ Comb_t). Sec. 3.2: the Evaluator
 * keeps a *payoff table* with one entry per combination, which a PSRO-style
 * meta-solver consumes; Sec. 4.2 estimates each entry by Monte-Carlo
 * simulations of the combination.
 *
 * Conventions for every call:
 *  - Return value: MALIB_OK (0) or a negative malib_status. No exception
 *    crosses this boundary. malib_last_error() gives a message for the last
 *    failing call on a context.
 *  - Pointers: "device" means memory of the context's GPU (cudaMalloc /
 *    torch tensors); "host or device" pointers are classified with
 *    cudaPointerGetAttributes. The caller owns every buffer it passes; the
 *    library keeps no pointer after the call's work has completed on the
 *    context's stream.
 *  - Ordering: calls are asynchronous and ordered on the context's CUDA stream,
 *    except that a call given a HOST output buffer copies the result back and
 *    waits for the stream before returning. Errors detected on the device
 *    (an invalid policy id in a device-side pair table, an expired bounded
 *    wait) are reported by the next malib_sync().
 *  - Threads: one context must not be used from two threads at once.
 */
#ifndef MALIB_H
#define MALIB_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum malib_status {
    MALIB_OK = 0,
    MALIB_EINVAL = -1,        /* bad argument (null pointer, size, id, layout) */
    MALIB_ENOMEM = -2,        /* device or host allocation failed */
    MALIB_ECUDA = -3,         /* a CUDA runtime call failed */
    MALIB_ESTATE = -4,        /* no population loaded, or env/population mismatch */
    MALIB_ETIMEOUT = -5,      /* a bounded device-side wait expired */
    MALIB_EUNSUPPORTED = -6,  /* valid request outside the built kernels' shapes */
    MALIB_ENOTCONVERGED = -7  /* an iterative solver reached its iteration limit */
} malib_status;

typedef enum malib_env_kind {
    MALIB_ENV_KUHN = 1,       /* Kuhn poker: 3 cards, ante 1, one bet of 1, 2 seats */
    MALIB_ENV_LEDUC = 2,      /* Leduc hold'em: 6 cards, 2 rounds, raises 2 then 4 */
    MALIB_ENV_SPREAD = 3,     /* cooperative particle spread (App. B.1) */
    MALIB_ENV_ADVERSARY = 4,  /* simple adversary (App. B.1): 1 adversary, 2 good agents */
    MALIB_ENV_SPEAKER_LISTENER = 5, /* simple speaker listener (App. B.1): speaker, listener */
    MALIB_ENV_PUSH = 6,       /* simple push (App. B.1): 1 adversary, 1 good agent, 1 landmark */
    MALIB_ENV_TAG = 7,        /* simple tag (App. B.1): 3 adversaries, 1 good agent, 2 obstacles */
    MALIB_ENV_REFERENCE = 8   /* simple reference (App. B.1): 2 agents that speak and move */
} malib_env_kind;

typedef enum malib_policy_kind {
    MALIB_POL_TABULAR = 1,    /* Kuhn: P(bet) for each of 6 infosets */
    MALIB_POL_MLP = 2         /* 3-layer ReLU MLP: in -> h1 -> h2 -> out logits */
} malib_policy_kind;

typedef enum malib_dtype {
    MALIB_F32 = 0,            /* fp32 weights, fp32 FMA forward */
    MALIB_BF16 = 1            /* bf16 weights and layer inputs, fp32 accumulation */
} malib_dtype;

/* Flags of malib_env_spec.flags and malib_eval_payoff_ex(). */
#define MALIB_DUMP_LOGITS 1u          /* record logits (and obs, actions) in a malib_traj */
#define MALIB_EXACT_EXPECTATION 2u    /* Kuhn: exact enumeration instead of Monte Carlo */
#define MALIB_SPREAD_LOCAL_RATIO 4u   /* SPREAD, REFERENCE: weight the reward terms by local_ratio */
#define MALIB_SPREAD_CONTACT 8u       /* SPREAD: agents push each other apart (contact forces) */

typedef struct malib_ctx malib_ctx;   /* opaque, library-owned */

/*
 * Environment description (the paper's env_desc, App. C.1 single-instance
 * example). Fixed shapes per kind:
 *   KUHN:   n_agents 2, obs_dim 0 (infoset index), n_actions 2
 *   LEDUC:  n_agents 2, obs_dim 17, n_actions 3 (fold, call/check, raise)
 *   SPREAD: n_agents = n_landmarks in [2, 16], obs_dim >= 4 + 4 n_agents - 2,
 *           n_actions 5 (noop, +x, -x, +y, -y), episode_len >= 1
 *   ADVERSARY: n_agents 3 (agent 0 the adversary, 1 and 2 the good agents),
 *           n_landmarks 2, obs_dim 14, n_actions 5, episode_len >= 1
 *   SPEAKER_LISTENER: n_agents 2 (agent 0 the speaker, 1 the listener),
 *           n_landmarks 3, obs_dim 11, n_actions 5, episode_len >= 1
 *   PUSH:   n_agents 2 (agent 0 the adversary, 1 the good agent),
 *           n_landmarks 1, obs_dim 8, n_actions 5, episode_len >= 1
 *   TAG:    n_agents 4 (agents 0..2 the adversaries, 3 the good agent),
 *           n_landmarks 2 (the obstacles), obs_dim 16, n_actions 5,
 *           episode_len >= 1
 *   REFERENCE: n_agents 2, n_landmarks 3, obs_dim 14, n_actions 15 (a = 5 *
 *           message + move), episode_len >= 1
 * n_envs is the number of parallel environments of a rollout (the particle
 * scenarios SPREAD, ADVERSARY, SPEAKER_LISTENER, PUSH, TAG, REFERENCE).
 * SPREAD reward of agent i after a step (App. B.1), with cover = sum over
 * landmarks of the distance to the nearest agent and coll_i = the number of
 * agents closer than 0.3 to agent i:
 *   default:                        r_i = -(cover + coll_i)
 *   flags & MALIB_SPREAD_LOCAL_RATIO: r_i = -((1 - local_ratio) cover + local_ratio coll_i)
 * (the paper's local_ratio, 0 <= local_ratio <= 1; each operation rounded in
 * fp32 in the order written).
 * ADVERSARY (App. B.1 simple adversary): the spread dynamics; at reset one of
 * the two landmarks is drawn as the target. With d(.) the distance to the
 * target after the step: adversary r_0 = -d(p_0); good agents r_1 = r_2 =
 * -min(d(p_1), d(p_2)) + d(p_0). Observation of agent i: velocity, position,
 * target - p_i (zeros for the adversary, which is not told the target), the two
 * landmarks - p_i, the other agents - p_i (ascending).
 * SPEAKER_LISTENER (App. B.1 simple speaker listener): at reset one of the
 * three landmarks is drawn as the target. The speaker does not move; its action
 * 0..2 is a message (actions 3 and 4 are never drawn for it). The listener
 * moves with the spread dynamics and observes the message sent at the previous
 * step. Both agents get r = -d(p_1, target) after the step. Observations (11
 * floats): speaker - one-hot of the target, zeros; listener - velocity, the
 * three landmarks - p_1, one-hot of the last message (zeros before the first).
 * Contact forces (App. B.1 names collisions and obstacles that block the way
 * but no force law; this is the soft contact model of the particle
 * environments): disks whose radii sum to dmin at distance d push each other
 * along the line of centres with force 100 * pen, pen = 0.001 * log(1 +
 * exp((dmin - d) / 0.001)), computed from the positions before the move and
 * added to the action forces. SPREAD with MALIB_SPREAD_CONTACT: the agents
 * (radius 0.15) push each other.
 * PUSH (App. B.1 simple push): agents of radius 0.15 that push each other, the
 * spread dynamics otherwise. With d_i = |p_i - landmark| after the step: good
 * agent r_1 = -d_1, adversary r_0 = d_1 - d_0. Observation of agent i (8
 * floats): velocity, position, landmark - p_i, the other agent - p_i.
 * TAG (App. B.1 simple tag): adversaries of radius 0.075 with action force 3
 * and speed limit 1.0, the good agent of radius 0.05 with action force 4 and
 * speed limit 1.3, immovable obstacles of radius 0.2; every agent pair and
 * every agent-obstacle pair collides. After the step an adversary hits the
 * good agent when closer than 0.125; with h hits, r_3 = -10 h and each
 * adversary gets 10 h. Observation of agent i (16 floats): velocity, position,
 * obstacles - p_i, the other agents - p_i (ascending), the good agent's
 * velocity for an adversary (zeros for the good agent).
 * REFERENCE (App. B.1 simple reference): at reset agent i's goal is one of the
 * three landmarks (chance draw with step field 0xC0000000 + i), told only to
 * the other agent. Action a moves by a % 5 (the spread dynamics, no contact)
 * and sends message a / 5 (0..2), which the other agent observes from the next
 * step on. With d_i = |p_i - goal_i| after the step and rho = local_ratio
 * (MALIB_SPREAD_LOCAL_RATIO; 0.5 without it): r_i = -((1 - rho) ((d_0 + d_1)
 * 0.5) + rho d_i). Observation of agent i (14 floats): velocity, the three
 * landmarks - p_i, the other agent's goal as a one-hot, the other agent's last
 * message as a one-hot (zeros before the first).
 */
typedef struct malib_env_spec {
    int32_t env_kind;
    int32_t n_agents;
    int32_t n_landmarks;
    int32_t obs_dim;
    int32_t n_actions;
    int32_t episode_len;
    int64_t n_envs;
    uint32_t flags;
    float local_ratio;        /* read only with MALIB_SPREAD_LOCAL_RATIO */
} malib_env_spec;

/*
 * One population member. params points to fp32 values (host or device) in the
 * layout
 *   TABULAR: p_bet[6], infoset index = card * 2 + h (card J=0, Q=1, K=2;
 *            h = 1 when facing a bet, where "bet" means call)
 *   MLP:     W1[h1][in], b1[h1], W2[h2][h1], b2[h2], W3[out][h2], b3[out]
 * nbytes must equal the byte size of that layout. dtype MALIB_BF16 rounds the
 * weights to bf16 (nearest-even) when loading; biases stay fp32.
 * seat: owning seat of a poker population (0 or 1), or -1 for a shared pool.
 */
typedef struct malib_policy_desc {
    int32_t kind;
    int32_t dtype;
    int32_t seat;
    int32_t n_layers;         /* 3 for MLP, 1 for TABULAR */
    int32_t dims[4];          /* MLP: in, h1, h2, out; TABULAR: 6, 0, 0, 1 */
    const void* params;
    int64_t nbytes;
} malib_policy_desc;

/*
 * Trajectory buffers, all DEVICE pointers, caller-owned, 16-byte aligned.
 * Rollout (SPREAD), T = episode_len, E = n_episodes per env, V = n_envs,
 * N = n_agents, P4 = obs_dim rounded up to a multiple of 4:
 *   obs     float [E][T][V][N][P4]  (padding columns are written as 0)
 *   action  uint8 [E][T][V][N]
 *   reward  float [E][T][V][N]
 *   done    uint8 [E][T][V]         (1 at t = T-1)
 *   logits  float [E][T][V][N][A]   (only with MALIB_DUMP_LOGITS; else may be NULL)
 * Evaluation dump (malib_eval_payoff_ex), first n_dump episodes of every pair,
 * S = max decisions per episode (Kuhn 3, Leduc 8), steps after the end padded:
 *   obs     float [n_pairs][n_dump][S][P4]  (Leduc 17 -> 20; Kuhn: unused)
 *   action  uint8 [n_pairs][n_dump][S]      (255 after the end)
 *   reward  float [n_pairs][n_dump][S]      (seat-0 payoff at the final decision, else 0)
 *   done    uint8 [n_pairs][n_dump][S]      (1 from the final decision on)
 *   logits  float [n_pairs][n_dump][S][A]   (Kuhn: A = 2, [1 - P(bet), P(bet)])
 * Any of the eval-dump pointers may be NULL to skip that field.
 */
typedef struct malib_traj {
    float* obs;
    uint8_t* action;
    float* reward;
    uint8_t* done;
    float* logits;
} malib_traj;

/* Creates a context on CUDA device `device`, ordered on `cuda_stream`
 * (a cudaStream_t; NULL = the legacy default stream). *out receives the
 * context; on failure *out is NULL. */
int malib_create(malib_ctx** out, int device, void* cuda_stream);

/* Frees the context, its population arena and scratch. Waits for the stream. */
void malib_destroy(malib_ctx* ctx);

/* Message of the last failing call on ctx ("" if none). Valid until the next
 * call on ctx. ctx may be NULL (message of the last failed malib_create). */
const char* malib_last_error(const malib_ctx* ctx);

/* Waits for the context's stream; returns deferred device-side errors
 * (MALIB_EINVAL for an invalid device pair table, MALIB_ETIMEOUT) and clears them. */
int malib_sync(malib_ctx* ctx);

/* Replaces the stream further calls are ordered on. */
int malib_set_stream(malib_ctx* ctx, void* cuda_stream);

/*
 * malib_pop_load - add policies to the population (Sec. 3.1: policy pools
 * P = {P_i}, extended as PSRO adds best responses, App. C.2 main loop).
 * Copies and converts the parameters into the context's device arena: the
 * plain fp32 parameters (host or device memory) are copied into a device
 * staging buffer and one kernel writes every policy's kernel image (fp32
 * layout, bf16-rounded weights, or the bf16 tensor-core image). The call waits
 * for its copies and the conversion on the context's stream, so the caller may
 * free `pols[i].params` when it returns. All policies of one
 * context share env kind, kind, dtype and dims; the first call fixes them and
 * `spec`. ids_out[n] receives the new policies' ids (consecutive, from 0).
 * Errors: EINVAL (shape or size mismatch with spec), ESTATE (different spec
 * than the loaded population), ENOMEM, ECUDA.
 */
int malib_pop_load(malib_ctx* ctx, const malib_env_spec* spec, const malib_policy_desc* pols,
                   int32_t n, int32_t* ids_out);

/* Drops the whole population (ids restart at 0). */
int malib_pop_reset(malib_ctx* ctx);

/*
 * malib_rollout - batched multi-agent rollout (Sec. 3.1, X(theta) ~ P(s, a, s'
 * | a ~ Comb_t); the Actor with k environments of the architecture figure).
 * SPREAD, ADVERSARY, SPEAKER_LISTENER, PUSH, TAG and REFERENCE (App. B.1
 * particle scenarios). Kernels: SPREAD N = 8 (obs 34, bf16 34-256-256-5 policies) on
 * the tensor cores; SPREAD N = 3 (obs 18) and the other scenarios with fp32
 * MLPs of hidden width 64, at most 128 environments per combination.
 * pair_ids (host or device) int32 [n_pairs][n_agents] holds one
 * policy id per agent for each combination; the n_envs environments are split
 * evenly and contiguously over the combinations (n_envs % n_pairs == 0).
 * Environment v of episode e uses global episode id g = e * n_envs + v; all
 * randomness is Philox4x32-10 keyed by seed with counter (g, step, agent).
 * traj_out (device buffers of the context's device, layout above) receives
 * n_episodes episodes per env. A device pair table or output on another GPU
 * gives EINVAL.
 * Errors: EINVAL, ESTATE, EUNSUPPORTED (a policy shape without a kernel).
 */
int malib_rollout(malib_ctx* ctx, const malib_env_spec* spec, const int32_t* pair_ids,
                  int32_t n_pairs, int64_t n_episodes, uint64_t seed, malib_traj* traj_out);

/*
 * malib_eval_payoff - empirical payoff table (Sec. 3.2 Evaluator; Sec. 4.2,
 * Monte-Carlo simulations per policy combination). KUHN and LEDUC.
 * pair_ids (host or device) int32 [n_pairs][2] = (seat-0 policy id, seat-1
 * policy id). Pair k plays n_episodes >= 1 hands with global episode ids
 * g = k * n_episodes + e. payoff_out (host or device) double [n_pairs][4]
 * receives, for the seat-0 payoff (seat 1 gets its negation):
 *   mean, standard error of the mean (sample variance / n, 0 if n < 2),
 *   sum, sum of squares (exact integers).
 * n_pairs == 0 is a no-op. Device buffers must belong to the context's device
 * (EINVAL otherwise). Errors: EINVAL, ESTATE, EUNSUPPORTED.
 */
int malib_eval_payoff(malib_ctx* ctx, const int32_t* pair_ids, int32_t n_pairs,
                      int64_t n_episodes, uint64_t seed, double* payoff_out);

/*
 * malib_eval_payoff_ex - malib_eval_payoff with flags:
 *   MALIB_DUMP_LOGITS: record the first n_dump (<= n_episodes) episodes of
 *     every pair into `dump` (device buffers, eval-dump layout above);
 *   MALIB_EXACT_EXPECTATION (KUHN): the entry's mean is the exact expected
 *     payoff by enumeration of the 6 deals; SE, sum and sum of squares are 0
 *     and n_episodes and seed are ignored.
 */
int malib_eval_payoff_ex(malib_ctx* ctx, const int32_t* pair_ids, int32_t n_pairs,
                         int64_t n_episodes, uint64_t seed, uint32_t flags, double* payoff_out,
                         const malib_traj* dump, int64_t n_dump);

/*
 * malib_eval_payoff_noalloc - malib_eval_payoff for callers that cannot
 * allocate device memory during the call. The paper has no counterpart; this is
 * a deployment variant. Typical callers: a framework that has already
 * reserved the GPU's memory in its own caching pool, or a latency-critical loop
 * in which cudaMalloc/cudaFree would synchronise the device and stall other
 * streams. This call allocates nothing: it calls no cudaMalloc, cudaFree or
 * allocating library routine. Its scratch (per-pair payoff sums, a decision
 * counter and per-pair hand counters) is a fixed file-scope device array of
 * 192 KiB + 8 B that every GPU loading the library holds until the process
 * exits.
 *  - pair_ids and payoff_out must be DEVICE buffers of the context's device
 *    (layouts as in malib_eval_payoff; no host staging). Host buffers, or
 *    buffers on another GPU, give EINVAL.
 *  - n_pairs <= 8192 (the array's capacity); more gives EINVAL.
 *  - The population must already be loaded (malib_pop_load), MC mode only,
 *    no dump. Kuhn populations and fp32 Leduc populations are served, with the
 *    same results as malib_eval_payoff for the same arguments; bf16 Leduc
 *    populations (tensor-core images) give MALIB_EUNSUPPORTED.
 *    malib_eval_stats does not report its decision count.
 *  - The first call on a device looks the array's device address up
 *    (cudaGetSymbolAddress); make that first call before any stream capture.
 *  - Every call shares the array and clears it first; calls that overlap on
 *    the GPU (other streams or contexts on the same device) race on it.
 */
int malib_eval_payoff_noalloc(malib_ctx* ctx, const int32_t* pair_ids, int32_t n_pairs,
                              int64_t n_episodes, uint64_t seed, double* payoff_out);

/* ---- meta-game solvers on payoff tables (Sec. 4.2, App. C.2) ----
 *
 * The PSRO loop of Sec. 4.2 turns the payoff table into a meta-strategy with a
 * meta-solver (fictitious play; an exact LP solver is named as the
 * alternative), and the training-loop listing of App. C.2 aggregates payoffs
 * under that equilibrium. These calls solve G zero-sum matrix games at once,
 * one CTA per game.
 *
 * Payoff layout (all calls): device fp64; element (g, i, j), seat 0's payoff
 * when row policy i meets column policy j, is payoff[((g*m + i)*n + j)*stride].
 * stride 1 reads a plain [G][m][n] table; stride 4 reads the mean column of
 * malib_eval_payoff's [n_pairs][4] output when its pairs are the row-major
 * Cartesian product of m rows and n columns. Entries must be finite.
 * All outputs are caller-owned device fp64 buffers. Calls are asynchronous on
 * the context's stream; EINVAL for host pointers or bad sizes, EUNSUPPORTED
 * for dimensions above the stated limits. The context needs no population.
 */

/* Fictitious play: both seats play policy 0 first, then each plays the first
 * (lowest-index) best response to the other's empirical play so far; the
 * cumulative payoffs are fp64 sums in play order, so results are reproducible
 * bit for bit. After iters >= 1 plays: x_out [G][m] and y_out [G][n] are the
 * empirical mixtures (play counts / iters); bounds_out [G][2] = {min_j (x^T
 * A)_j, max_i (A y)_i}, which bracket the game value (their difference is the
 * mixtures' NashConv). 1 <= m, n <= 1024. */
int malib_meta_fictitious_play(malib_ctx* ctx, const double* payoff, int32_t n_games, int32_t m,
                               int32_t n, int32_t stride, int64_t iters, double* x_out,
                               double* y_out, double* bounds_out);

/* Exact equilibrium by linear programming (simplex, Bland's rule): value_out
 * [G] = the game value; x_out [G][m], y_out [G][n] one equilibrium (not unique
 * in general). 1 <= m, n <= 512; tableaus larger than 200 KB live in
 * context-owned device memory. A game that reaches the pivot limit raises
 * MALIB_ENOTCONVERGED at the next malib_sync. */
int malib_meta_lp_nash(malib_ctx* ctx, const double* payoff, int32_t n_games, int32_t m,
                       int32_t n, int32_t stride, double* x_out, double* y_out,
                       double* value_out);

/* malib_meta_lp_nash with the pivot limit chosen by the caller: max_pivots > 0
 * caps the pivots of every game at that number; 0 keeps the default limit of
 * 50 (m + n) + 1000. A game that needs more pivots than the limit leaves its
 * outputs at the last tableau (not an equilibrium) and raises
 * MALIB_ENOTCONVERGED at the next malib_sync, which clears it; the context
 * stays usable. EINVAL for max_pivots < 0. */
int malib_meta_lp_nash_ex(malib_ctx* ctx, const double* payoff, int32_t n_games, int32_t m,
                          int32_t n, int32_t stride, int32_t max_pivots, double* x_out,
                          double* y_out, double* value_out);

/* Payoffs under mixtures x [G][m], y [G][n] (device fp64): row_payoff_out
 * [G][m] = A y (what each row policy, e.g. a new best response, earns against
 * the column mixture), col_payoff_out [G][n] = x^T A, value_out [G] = x^T A y
 * (the equilibrium's expected payoff). */
int malib_meta_aggregate(malib_ctx* ctx, const double* payoff, int32_t n_games, int32_t m,
                         int32_t n, int32_t stride, const double* x, const double* y,
                         double* row_payoff_out, double* col_payoff_out, double* value_out);

/* Exploitability of a pair of seat mixtures (Sec. 4.2: PSRO's convergence is
 * measured by exploitability). ids0 [n0] are seat-0 policy ids of the loaded
 * population with weights x [n0], ids1 [n1] seat-1 ids with weights y [n1]
 * (fp64; normally each sums to 1, e.g. a fictitious-play or LP mixture).
 * out [3] = {b0, b1, (b0 + b1) / 2}: b0 is the best seat-0 strategy's expected
 * payoff against the seat-1 mixture, b1 the best seat-1 strategy's against the
 * seat-0 mixture; a best responder sees its card, the public card once dealt
 * and the betting history. Kuhn (tabular) and Leduc (MLP 17-h1-h2-3 fp32 with
 * h <= 256, or bf16 17-256-256-3) populations; 1 <= n0, n1 <= 256. Policy
 * action probabilities: the fp64 softmax, over legal actions, of the logits of
 * the policy's forward (fp32 FMA; bf16 operands for bf16 policies).
 * Arguments may be host or device memory; the call waits for the result. */
int malib_exploitability(malib_ctx* ctx, const int32_t* ids0, const double* x, int32_t n0,
                         const int32_t* ids1, const double* y, int32_t n1, double* out);

/* ---- learner side: the next stage of the loop, consuming traj_out ---- */

/*
 * malib_learn_pg - one independent learner's policy-gradient step (Sec. 3.3
 * "Independent Learning": one learner per policy, trained on its own agents'
 * experience; App. C.2: the training workflow samples rollout episodes into a
 * batch for the learner's optimize()). For policy `policy_id` its samples S
 * are every (episode, step, environment, agent) of the rollout in traj whose
 * combination (pair_ids [n_pairs][n_agents], host or device, the table the
 * rollout used) gives that agent policy_id; M = |S|. With G the discounted
 * return-to-go of a sample within its episode (G_t = r_t + gamma G_{t+1}),
 * b the mean of G over S and H the entropy of the policy's softmax over the
 * 5 actions, the loss is
 *   L = -(1/M) sum_S [ (G - b) log pi(a | o) + entropy_coef H(pi(. | o)) ]
 * and grad_out (host or device, float [P]) receives dL/dparams in the
 * malib_policy_desc parameter layout (W1, b1, W2, b2, W3, b3; P parameters).
 * stats_out (optional, host or device, double [4]) receives M, b, L and the
 * mean entropy. traj: obs, action and reward of malib_rollout (device memory
 * of the context's device, the rollout's spec, n_episodes and episode_len).
 * Built for particle-scenario populations of fp32 MLPs in-64-64-5 with in
 * <= 32 (EUNSUPPORTED otherwise); gamma in [0, 1], entropy_coef >= 0.
 * Deterministic (fixed-order sums, no atomics). Waits for the stream before
 * returning. Errors: EINVAL, ESTATE, EUNSUPPORTED.
 */
int malib_learn_pg(malib_ctx* ctx, const malib_env_spec* spec, const int32_t* pair_ids, int32_t n_pairs,
                   int64_t n_episodes, const malib_traj* traj, int32_t policy_id, float gamma,
                   float entropy_coef, float* grad_out, double* stats_out);

/*
 * malib_learn_pg_batch - malib_learn_pg for n_policies distinct policies at
 * once, each its own independent learner (Sec. 3.3), in one launch sequence:
 * policy_ids (host) int32 [n_policies], grad_out (host or device) float
 * [n_policies][P], stats_out (optional, host or device) double
 * [n_policies][4], each row malib_learn_pg's for that policy up to the
 * rounding of its sums (a batch shares the policies' tiles among the CTAs
 * differently; a given batch is deterministic). A repeated id gives EINVAL. Waits for the stream before returning. Errors: EINVAL,
 * ESTATE, EUNSUPPORTED.
 */
int malib_learn_pg_batch(malib_ctx* ctx, const malib_env_spec* spec, const int32_t* pair_ids, int32_t n_pairs,
                         int64_t n_episodes, const malib_traj* traj, const int32_t* policy_ids,
                         int32_t n_policies, float gamma, float entropy_coef, float* grad_out,
                         double* stats_out);

/*
 * malib_learn_ppo_batch - malib_learn_pg_batch with PPO's clipped surrogate
 * (Schulman et al. 2017; the paper's learners are PPO/A2C-style, Sec. 3.3 and
 * App. C.2) in place of (G - b) log pi(a | o): with A = G - b as above and
 * rho = pi(a | o) / mu(a | o), mu the behavior policy that acted in the rollout,
 *   L = -(1/M) sum_S [ min(rho A, clip(rho, 1 - clip_eps, 1 + clip_eps) A)
 *                      + entropy_coef H(pi(. | o)) ].
 * mu is read from traj->logits, the logits [n_episodes][T][n_envs][N][5] that
 * malib_rollout recorded under MALIB_DUMP_LOGITS (device memory of the
 * context's device; EINVAL when NULL); pi is the loaded policy, so after
 * malib_pop_update the same samples give the next epoch's gradient. Where the
 * unclipped term is the minimum (ties included) it carries the gradient
 * A rho (pi - onehot(a)) / M at the logits; elsewhere the surrogate is constant.
 * With the loaded policy equal to the behavior policy (rho = 1) the gradient
 * is malib_learn_pg_batch's up to rounding. clip_eps in (0, 1). Rows of
 * grad_out and stats_out as in malib_learn_pg_batch (stats: M, b, L, mean
 * entropy). Waits for the stream before returning. Errors: EINVAL, ESTATE,
 * EUNSUPPORTED.
 */
int malib_learn_ppo_batch(malib_ctx* ctx, const malib_env_spec* spec, const int32_t* pair_ids, int32_t n_pairs,
                          int64_t n_episodes, const malib_traj* traj, const int32_t* policy_ids,
                          int32_t n_policies, float gamma, float entropy_coef, float clip_eps, float* grad_out,
                          double* stats_out);

/*
 * malib_adam_step - one Adam step (the optimizer of App. C.2's training
 * config; Kingma and Ba, with bias correction) on n parameters, in place:
 *   m <- beta1 m + (1 - beta1) g;  v <- beta2 v + (1 - beta2) g^2;
 *   params <- params - lr (m / (1 - beta1^step)) / (sqrt(v / (1 - beta2^step)) + eps).
 * params, grad, m, v: float [n] device buffers of the context's device (the
 * caller owns them; m and v start at zero). step >= 1 counts the calls.
 * Asynchronous on the context's stream. Errors: EINVAL.
 */
int malib_adam_step(malib_ctx* ctx, float* params, const float* grad, float* m, float* v, int64_t n,
                    int64_t step, float lr, float beta1, float beta2, float eps);

/*
 * malib_pop_update - replaces the parameters of loaded policy `policy_id`
 * (Sec. 3.1: the learner's new policy goes back into the population that the
 * next rollouts and evaluations use). params: host or device, the
 * malib_policy_desc layout of the policy's shape, nbytes its size. The
 * policy's kernel image is rebuilt in place; work already queued on the
 * context's stream sees the old parameters. Returns once the caller's buffer
 * may be reused. Errors: EINVAL, ESTATE.
 */
int malib_pop_update(malib_ctx* ctx, int32_t policy_id, const float* params, int64_t nbytes);

/* ---- measurement and self-test entry points (used by tests and the benchmark) ---- */

/* Total decisions (env-steps: one decision by the acting seat) played by the
 * most recent Monte-Carlo malib_eval_payoff[_ex] call on ctx. Waits for the
 * stream. ESTATE if none has run. */
int malib_eval_stats(malib_ctx* ctx, int64_t* n_decisions);

/* Number of kernels this context has launched since creation. */
int64_t malib_launch_count(const malib_ctx* ctx);

/* Enables (1) or disables (0) CUDA-event timing of each call's main kernel on
 * the context's stream (for malib_learn_pg[_batch], the gradient kernel);
 * malib_main_kernel_ms() returns the summed milliseconds
 * of the timed launches since the last reset (waits for the stream) and the
 * number of launches timed in *n_launches (may be NULL); reset clears both. */
int malib_set_timing(malib_ctx* ctx, int enable);
double malib_main_kernel_ms(malib_ctx* ctx, int64_t* n_launches, int reset);

/* Philox4x32-10 of n counters (device uint32 [n][4]) under key (seed lo, seed
 * hi) into out (device uint32 [n][4]) - the generator every kernel draws from. */
int malib_selftest_philox(malib_ctx* ctx, const uint32_t* ctr, uint64_t seed, uint32_t* out,
                          int64_t n);

/* Philox4x32-10 digest (the generator of Sec. 3.1's sampled rollouts, keyed as
 * above): thread t < n XOR-folds the four output words of the calls
 * i = 0..calls-1 at counter (t lo32, t hi32, i, 0) under key (seed lo32, seed
 * hi32) into out[t] (device uint32 [n], caller-owned). Its work is generator
 * arithmetic only, so its rate (calls per second) is the ALU ceiling of the Kuhn
 * evaluation, whose per-hand work is Philox calls. EINVAL for n < 0, calls < 0
 * or a host pointer; asynchronous on the context's stream. */
int malib_philox_digest(malib_ctx* ctx, uint64_t seed, int64_t n, int32_t calls, uint32_t* out);

/* Bounded-wait self-test: one device thread waits at most limit_ns
 * (1 <= limit_ns <= 1e9) for an mbarrier phase; with arrive = 0 nothing
 * completes it, the wait expires and the kernel records a timeout, which the
 * next malib_sync reports as MALIB_ETIMEOUT (the context stays usable); with
 * arrive != 0 the thread completes the phase itself first and no error is
 * recorded. Every wait of the library's kernels is bounded the same way. */
int malib_selftest_wait(malib_ctx* ctx, int32_t arrive, int64_t limit_ns);

/* The kernels' deterministic exp (Cody-Waite reduction, degree-7 Taylor) on n
 * device floats, and the masked inverse-CDF draw on n rows of A <= 8 logits
 * (device: logits [n][A], legal uint8 [n][A], u [n], out int32 [n]). */
int malib_selftest_det_expf(malib_ctx* ctx, const float* x, float* y, int64_t n);
int malib_selftest_sample(malib_ctx* ctx, const float* logits, const uint8_t* legal,
                          const float* u, int32_t A, int32_t* out, int64_t n);

/* Tensor-core self-test: D[128][N] = A[128][K] . B[N][K]^T on one CTA with
 * tcgen05 MMAs from shared memory and an fp32 accumulator in tensor memory -
 * the operand layout and MMA path of the bf16 policy kernels. dtype MALIB_BF16:
 * A, B hold bf16 bit patterns (K % 16 == 0); MALIB_F32: A, B fp32, multiplied
 * as tf32 (K % 8 == 0). N % 16 == 0, 16 <= N <= 256; all device buffers,
 * row-major. */
int malib_selftest_mma(malib_ctx* ctx, int32_t dtype, const void* A, const void* B, float* D,
                       int32_t N, int32_t K);

/* Policy forward (Sec. 3.1: the policy's action distribution for an
 * observation; a3 of the rollout) on the pipelined tensor-core engine alone:
 * logits_out [n_rows][A] = the MLP of policy `policy_id` of the loaded bf16
 * population on the fp32 observation rows x [n_rows][in] (bf16 weights and
 * layer inputs, fp32 accumulation; layer 3 on the CUDA cores). Built for the
 * 17-256-256-3 Leduc populations (observation feature 15 must be 1, as every
 * Leduc state has it) and 34-256-256-5 populations; other shapes give
 * EUNSUPPORTED. reps >= 1 repeats the whole set (the same logits are written
 * again) so that the engine's rate can be measured on resident inputs. x and
 * logits_out are device buffers of the context's device; asynchronous on the
 * context's stream. */
int malib_selftest_mlp_tc(malib_ctx* ctx, int32_t policy_id, const float* x, int64_t n_rows,
                          int32_t reps, float* logits_out);

#ifdef __cplusplus
}
#endif

#endif /* MALIB_H */
