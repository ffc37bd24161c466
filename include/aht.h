/*
 * aht.h -- C ABI of libaht.so, the GB300 (sm_103a) batched ad hoc teamwork rollout path.
 *
 * The operations follow the paper "JaxAHT: A JAX-Based Library for Ad Hoc Teamwork":
 *   - the Dec-POMDP M = <S, {A_i}, P, {O_i}, Omega, r, rho, gamma> of Sec. 3 (joint
 *     action -> next state, per-agent observation, one shared team reward), stepped for
 *     thousands of independent envs at once (Sec. 5.1: the speedup comes from massive
 *     env parallelism);
 *   - an ego policy pi_e and teammates pi_{-e} drawn from a population (Sec. 3,
 *     T_train / T_eval), both decentralised MLP policies pi_i(a | o_i);
 *   - PPO rollout collection with GAE targets (App. C, "PPO ego");
 *   - the ego-by-teammate cross-play (XP) return matrix (App. B, "Cross-play matrix
 *     construction"); its row mean over held-out teammates is J_AHT of Sec. 3.
 * The paper does not state the game rules; the library implements readings of the
 * workload descriptions, stated rule by rule in the env sources (csrc/env_*.cuh) and in
 * the test oracle's header.
 *
 * Conventions (all entry points):
 *   - Bulk tensors are DEVICE pointers owned by the caller, laid out as documented,
 *     and must stay valid until the work enqueued on the context's stream completes.
 *     Small id lists (ego/teammate ids, teammate pools) are HOST arrays, passed by value
 *     to the kernels.
 *   - Calls are asynchronous on the CUDA stream given to aht_create (NULL = legacy
 *     default stream), except aht_create, aht_destroy, aht_get_state, aht_set_state and
 *     aht_sync, which synchronise that stream.
 *   - Host-side argument errors are returned immediately (AHT_EINVAL) and nothing is
 *     enqueued.  Errors detected on the device (an out-of-range id, an illegal forced
 *     Hanabi action, a wait of a tensor-core kernel that ran past its time limit) are
 *     latched in a device status word and returned by aht_sync.
 *   - Every wait of a kernel on another warp's progress (mbarriers, named barriers fed
 *     by them) is bounded by %globaltimer, 2 s by default: on expiry the kernel latches
 *     the timeout bit, stops its work, drains its own tensor-core operations and copies,
 *     frees its tensor memory and returns, so the context stays usable.
 *   - Only aht_create allocates device memory.  Every other call allocates nothing.
 *   - Seat 0 is the ego, seat 1 the teammate.  XP matrices are [ego][teammate]
 *     (the transpose of the paper's figures, whose rows are teammates).
 *   - Randomness is Philox4x32-10 (Salmon et al., SC'11), key = (seed lo, seed hi),
 *     counter = (env, step, stream, block); streams 0/1 = action of seat 0/1, 2 = env
 *     reset, 3 = teammate assignment.  "step" is the context's global step counter.
 *   - aht_last_error returns a thread-local message for the last failing call.
 */
#ifndef AHT_H
#define AHT_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct aht_ctx aht_ctx; /* opaque, library-owned */

typedef enum aht_status {
  AHT_OK = 0,
  AHT_EINVAL = 1,   /* invalid argument (host check) */
  AHT_ENOMEM = 2,   /* device allocation failed in aht_create */
  AHT_ECUDA = 3,    /* a CUDA runtime call failed */
  AHT_ETIMEOUT = 4, /* a bounded device wait gave up (reported by aht_sync) */
  AHT_EDEVICE = 5   /* the device status word recorded an error */
} aht_status;

enum { AHT_LBF = 0, AHT_OVERCOOKED = 1, AHT_HANABI = 2, AHT_MINI_HANABI = 3 };
enum { AHT_FP32 = 0, AHT_BF16 = 1 };

/* Environment (Sec. 4, Table "JaxAHT Environments"; the Dec-POMDP of Sec. 3).
 *   LBF: width, height in 3..12; n_food 1..3; agent levels uniform in 1..max_agent_level
 *        (1..9); episode_len >= 1.  Obs = width*height*4 u8, actions 6.
 *   Overcooked: the fixed 5x4 kitchen (width 5, height 4); episode_len >= 1;
 *        cook_time 0..255; soup_reward.  Obs = 520 u8, actions 6.
 *   Hanabi: 2 players, full deck; episode_len must be 0 (run to termination; a game
 *        lasts at most 97 turns, the library stops any game at 100).  Obs = 660 u8,
 *        actions 20 with illegal-action masking.
 *   Mini Hanabi (Sec. 4 Table: 3 colours x 3 ranks): 2 players, ranks 1,1,1,2,2,3 per
 *        colour (18 cards), 2-card hands, 3 info and 1 life tokens; episode_len must be
 *        0.  Obs = 156 u8 (153 features + 3 zero), actions 10 (play slot 0-1, discard
 *        slot 0-1, hint colour 0-2, hint rank 1-3) with illegal-action masking. */
typedef struct aht_env_desc {
  int32_t kind;
  int32_t width, height;
  int32_t n_food;
  int32_t max_agent_level;
  int32_t episode_len;
  int32_t cook_time, soup_reward;
} aht_env_desc;

/* Population of MLP policies (Sec. 3 pi_i; App. C: the ego and the teammates it meets).
 * Every policy is z = W3 tanh(W2 tanh(W1 o + b1) + b2) + b3 with
 *   W1 [hidden0][obs_dim], W2 [hidden1][hidden0], W3 [n_out_p][hidden1], row-major,
 *   b1 [hidden0], b2 [hidden1], b3 [n_out_p],
 * n_out_p = n_actions + has_value_head[p]: the optional last row is a value estimate.
 * W[3*p + l] / b[3*p + l] point at layer l of policy p, host or device memory, of
 * weight_dtype (fp32 or bf16).  aht_create copies and packs them; the caller may free
 * them afterwards.  has_value_head may be NULL (no value rows).
 * Limits: n_policies 1..1024, obs_dim must equal the env's, hidden0/hidden1 multiples
 * of 16 in 16..512. */
typedef struct aht_pop_desc {
  int32_t n_policies;
  int32_t obs_dim, hidden0, hidden1, n_actions;
  const int32_t* has_value_head; /* host [n_policies] of 0/1, or NULL */
  int32_t weight_dtype;          /* AHT_FP32 or AHT_BF16 */
  const void* const* W;          /* host array of 3*n_policies pointers */
  const void* const* b;          /* host array of 3*n_policies pointers */
} aht_pop_desc;

/* Rule-based LBF teammates (App. F, LBF heuristic suite).  A teammate id -1 - k in a
 * pool (aht_rollout) or teammate list (aht_xplay_matrix, aht_xplay_matrix_static) of an
 * LBF context whose policies run on the tensor-core path (hidden widths 64 or 128,
 * obs_dim <= 255, at most 7 actions + value; fp32 or bf16) selects heuristic k instead of
 * a network (other contexts return AHT_EINVAL for negative ids):
 *   k 0..4  Greedy: the uneaten food with the least distance to itself | distance to the
 *           ego | sum of the two | level | the greatest level (ties: lower food index);
 *   k 5..10 Sequential: the first uneaten food in the order of row-major cell index
 *           (y*width + x) ascending | descending, column-major index (x*height + y)
 *           ascending | descending, distance from its own position at the episode's start
 *           ascending | descending (ties: lower food index);
 *           then: load when 4-adjacent to it;
 *   k 11    Entitled: the pair of squares of the lowest-index uneaten food is its first
 *           two neighbours in the order W, E, N, S that lie on the grid and hold no
 *           uneaten food (fewer than two: noop); noop until the ego stands on one of them,
 *           then it goes for the other and loads when standing on it;
 * a move is one step along the axis with the larger remaining distance (ties: x), or
 * along the other axis when that cell is off the grid, an uneaten food or the ego; else
 * noop (distances Manhattan).  The rule draws nothing; the teammate's recorded action is
 * the rule's.  The paper names the criteria and orderings only: the rules above are this
 * library's reading. */
#define AHT_LBF_N_HEURISTICS 12
#define AHT_LBF_HEURISTIC(k) (-1 - (k))

/* Creates a context for up to n_envs concurrent envs (1 <= n_envs <= 2^30; PPO state and
 * cross-play batch capacity), packs the population and resets every env with `seed`
 * (step counter 0).
 * cuda_stream is a cudaStream_t (NULL = default stream).  Allocates all device memory
 * the context will ever use.  Returns AHT_EINVAL, AHT_ENOMEM or AHT_ECUDA on failure
 * (*out is then NULL). */
aht_status aht_create(const aht_env_desc* env, const aht_pop_desc* pop, int64_t n_envs,
                      uint64_t seed, void* cuda_stream, aht_ctx** out);
void aht_destroy(aht_ctx* ctx);

/* rho of Sec. 3: re-draws the initial state of all n_envs envs with a new seed and
 * sets the global step counter to 0.  Env e uses counter (e, 0, stream 2). */
aht_status aht_reset(aht_ctx* ctx, uint64_t seed);

/* Trajectory buffers of aht_rollout: caller-owned device memory, time-major [T][N]
 * (N = the context's n_envs).  NULL members are not written. */
typedef struct aht_traj {
  uint8_t* obs;         /* [T][N][obs_dim] ego observation before each step */
  uint8_t* actions;     /* [T][N] ego action */
  uint8_t* tm_actions;  /* [T][N] teammate action */
  float* logp;          /* [T][N] log pi_e(a | o) of the ego action */
  float* values;        /* [T][N] ego value (0 if the ego has no value row) */
  float* rewards;       /* [T][N] shared team reward r_t */
  uint8_t* dones;       /* [T][N] 1 if step t ended the episode (auto-reset follows) */
  float* advantages;    /* [T][N] GAE advantage */
  float* targets;       /* [T][N] advantage + value */
  float* last_value;    /* [N] value of the state after step T-1 (the bootstrap V_T) */
  int32_t* teammate;    /* [N] teammate policy id used by each env in this call */
  float gamma, lambda;  /* GAE discount and trace parameters, in [0, 1] */
} aht_traj;

/* PPO rollout collection (App. C "PPO ego"; Sec. 3 ego vs teammates from T_train).
 * Every env draws its teammate once per call: env e plays pool[floor(x * pool_size /
 * 2^32)] with x the first draw of counter (e, step0, stream 3), and keeps it for the
 * whole call, auto-reset episodes included, so each env meets a uniformly drawn pool
 * member, independently of its neighbours.  The envs are grouped by their draw so that a
 * tensor-core tile runs one teammate policy (the tiles of a group are not contiguous env
 * ranges; a pool of p members makes at most ceil(n_envs / 128) + p tiles).  Then for t in
 * 0..T-1 (step step0+t): both seats observe, the ego and the teammate MLPs run, actions
 * are sampled by inverse CDF with u from stream 0/1, the env steps, and an env whose
 * episode ended is reset at step step0+t+1 (stream 2).  Finally V_T is computed and GAE
 * (advantages, targets) is formed when `advantages` is non-NULL.  The step counter
 * advances by T.  Simultaneous-move envs only (LBF, Overcooked): AHT_EINVAL for Hanabi.
 * pool: host [pool_size] policy ids, 1 <= pool_size <= 256 (ids may repeat; each entry is
 * drawn with probability 1 / pool_size).  out->obs must be 4-byte aligned when
 * pool_size > 1.  T >= 1. */
aht_status aht_rollout(aht_ctx* ctx, int32_t ego_id, const int32_t* pool, int32_t pool_size,
                       int32_t T, const aht_traj* out);

/* PPO collection with per-episode teammates (Sec. 3: every episode pairs the ego with a
 * teammate drawn from the training set).  The episode of env e that began at step s
 * plays pool[floor(x * pool_size / 2^32)], x the first draw of counter (e, s, stream 5);
 * the context carries per env the step its current episode began (aht_reset: 0; every
 * auto-reset at step s' -- in any collection call or aht_step_forced -- sets s'; part of
 * the checkpoint).  Each step regroups the envs by teammate, so this call runs one launch
 * per step instead of one per call (on the tensor-core path each step's launch groups
 * its own rows and starts while the step before finishes; on the CUDA-core path a
 * grouping launch precedes each step's launch); otherwise the step, the draws and the
 * trajectory layout are those of aht_rollout.  out->teammate receives the teammate of the call's first step; teammates
 * (device int32 [T][N], or NULL) the teammate of every step.  out->obs must be 4-byte
 * aligned.  Same pool rules as aht_rollout (rule teammates on LBF tensor-core contexts). */
aht_status aht_rollout_resample(aht_ctx* ctx, int32_t ego_id, const int32_t* pool,
                                int32_t pool_size, int32_t T, const aht_traj* out,
                                int32_t* teammates);

/* IPPO collection (Sec. 3, the MARL baseline IPPO: both seats learn, each with its own
 * PPO of App. C).  Every env pairs policy0 in seat 0 with policy1 in seat 1; the call is
 * aht_rollout(ctx, policy0, {policy1}, 1, T, out0) -- the same draws, states and seat-0
 * trajectory -- and it also writes seat 1's learner trajectory to out1, in the layout
 * of aht_traj: obs = seat 1's observation (4-byte aligned), actions = seat 1's action,
 * tm_actions = seat 0's, logp / values / last_value of policy1 (values 0 without its
 * value row), the shared team reward, dones, and GAE into out1's advantages / targets
 * when those are non-NULL.  out1->teammate is not written.  policy1 is a network
 * (0 <= policy1 < n_policies); a trajectory of out1 is an aht_ppo_update input for a
 * learner of policy1. */
aht_status aht_rollout_ippo(aht_ctx* ctx, int32_t policy0, int32_t policy1, int32_t T,
                            const aht_traj* out0, const aht_traj* out1);

/* Outputs of aht_xplay_matrix (caller-owned device memory; NULL members not written). */
typedef struct aht_xplay_out {
  float* matrix;        /* [n_ego][n_tm] mean team return over the pair's envs */
  float* returns;       /* [n_ego][n_tm][P] team return of each env's first episode */
  int32_t* steps;       /* [n_ego][n_tm][P] env-steps the episode took */
  uint8_t* actions;     /* [max_steps][n_ego*n_tm*P][2] applied actions, 255 = none */
} aht_xplay_out;

/* Cross-play evaluation (App. B; J_AHT of Sec. 3 is a row mean).  Pair (i, j) plays
 * P = envs_per_pair fresh episodes of ego_ids[i] (seat 0) with tm_ids[j] (seat 1); env
 * index e = (i*n_tm + j)*P + k is reset at counter (e, step0, stream 2) and steps at
 * step0 + s.  An env stops after its first episode.  matrix[i][j] = (sum of the P fp32
 * returns, added exactly in fp64) / P.  Uses the context's scratch, not its PPO env
 * state; the step counter advances by max_steps.  Requires n_ego*n_tm*P <= n_envs,
 * 1 <= n_ego, n_tm <= 64, max_steps >= 1.  ego_ids / tm_ids are host arrays. */
aht_status aht_xplay_matrix(aht_ctx* ctx, const int32_t* ego_ids, int32_t n_ego,
                            const int32_t* tm_ids, int32_t n_tm, int32_t envs_per_pair,
                            int32_t max_steps, const aht_xplay_out* out);

/* Cross-play matrix that needs no device memory beyond its output (the paper has no
 * counterpart; this is a deployment convenience).  aht_xplay_matrix keeps the per-env
 * returns in context scratch sized at aht_create, so its batch is capped by the
 * context's n_envs; a caller that cannot allocate more device memory after start-up
 * (a host whose allocator is owned by another framework, or a long-lived PPO context
 * created with only its training batch) cannot grow that scratch.  This variant keeps
 * the per-env returns in one file-scope device array of AHT_XPLAY_STATIC_MAX_ENVS
 * floats (256 KiB) instead, which every GPU that loads the library holds until the
 * process exits, so any n_ego*n_tm*envs_per_pair up to that maximum works on any
 * context.  Same semantics and step counter as aht_xplay_matrix with only `matrix`
 * requested (device f32 [n_ego][n_tm]), and the same result for LBF contexts; for bf16
 * Overcooked and Hanabi contexts aht_xplay_matrix runs a streamed tensor-core kernel
 * whose buffers are sized by the context, this variant the CUDA-core kernel, so an
 * action can differ where the sampling CDF lies within ~1e-6 of the draw.
 *   - Allocates nothing and calls no allocating CUDA or library routine.
 *   - Returns AHT_EINVAL if n_ego*n_tm*envs_per_pair > AHT_XPLAY_STATIC_MAX_ENVS.
 *   - The first call on each device looks up the array's device address (with that
 *     device current) and caches it; make that first call before any stream capture.
 *   - All calls, on every context and stream of a device, share the one array; each
 *     call writes every entry it reads before reading it, so nothing needs clearing, but
 *     calls that overlap on the GPU race and must be serialised by the caller.
 *   - When aht_sync reports AHT_ETIMEOUT for the call, the cells of the pairs whose
 *     tiles gave up hold NaN (their returns are written as NaN, never left stale). */
#define AHT_XPLAY_STATIC_MAX_ENVS 65536
aht_status aht_xplay_matrix_static(aht_ctx* ctx, const int32_t* ego_ids, int32_t n_ego,
                                   const int32_t* tm_ids, int32_t n_tm, int32_t envs_per_pair,
                                   int32_t max_steps, float* matrix);

/* Outputs of aht_xp_stats (caller-owned device memory; NULL members not written). */
typedef struct aht_xp_stats_out {
  float* norm;        /* [n_ego][n_tm] xp / upper, NaN where upper <= 0 */
  float* regret;      /* [n_ego][n_tm] upper - xp */
  float* j_aht;       /* [n_ego] mean of the row (J_AHT, teammates uniform) */
  float* j_norm;      /* [n_ego] mean of the row of norm (NaN if any bound <= 0) */
  float* max_regret;  /* [n_ego] largest regret of the row */
  int32_t* worst_tm;  /* [n_ego] its column (the lowest on ties) */
  float* brdiv;       /* [1] BRDiv cross-play objective; n_ego == n_tm only */
} aht_xp_stats_out;

/* What the evaluation and teammate-generation stages compute from a cross-play matrix
 * (device f32 [n_ego][n_tm], e.g. aht_xplay_matrix's; rows are the policies in the ego
 * seat -- best responses or the ego -- and columns the evaluation teammates):
 *   - upper (device f32 [n_tm], in/out): App. B "Upper bound estimation" -- each
 *     teammate's recorded best-response bound is replaced by any score of its column
 *     that exceeds it (strict >: pass -inf for "no bound yet"; a NaN bound stays NaN);
 *   - norm = xp / upper: the return relative to the best response's (Sec. 3, App. B
 *     "normalized return"), NaN where the bound is <= 0;
 *   - regret = upper - xp: App. A ROTATE's cooperative regret (best-response return minus
 *     the return achieved), max_regret / worst_tm its row maximum and that teammate;
 *   - j_aht: Sec. 3 J_AHT with the teammates weighted uniformly; j_norm the same of norm;
 *   - brdiv = mean of the diagonal - mean of the off-diagonal entries (App. A BRDiv:
 *     matched teammate/best-response returns high, mismatched cross-play low; unit
 *     weights, the off-diagonal term 0 for n = 1).
 * Arithmetic is fp64, each output rounded to f32 once; the elementwise outputs, bounds
 * and max_regret/worst_tm are exact, the means are sums in a fixed order (a warp per row,
 * lanes over every 32nd column, then a shuffle tree), deterministic from call to call and
 * within one f32 rounding of any other summation order.  One small kernel on
 * cuda_stream (a cudaStream_t, NULL = default stream); allocates nothing.
 * Returns AHT_EINVAL for NULL xp/upper/out, n_ego or n_tm outside 1..AHT_XP_STATS_MAX,
 * or brdiv requested for a non-square matrix. */
#define AHT_XP_STATS_MAX 2048
aht_status aht_xp_stats(const float* xp, int32_t n_ego, int32_t n_tm, float* upper,
                        const aht_xp_stats_out* out, void* cuda_stream);

/* ---- PPO ego update (App. C "PPO ego") ----------------------------------------------
 * The paper trains the ego with PPO (Schulman et al. 2017) against its teammates and
 * states no loss details; the update implemented is that paper's clipped surrogate:
 *   per sample  rho = exp(logp(a) - logp_old),  A_n = (A - mean_mb A) / (std_mb A + 1e-8),
 *   L = -min(rho A_n, clip(rho, 1 - clip_eps, 1 + clip_eps) A_n)
 *       + vf_coef * 0.5 max((V - R)^2, (V_old + clip(V - V_old, -clip_eps, clip_eps) - R)^2)
 *       - ent_coef * H(pi),
 * averaged over each minibatch (mean and population std of A over the minibatch, R the
 * targets); the gradient is clipped to global norm max_grad_norm (if > 0) and applied by
 * Adam (Kingma & Ba 2015; m_hat / (sqrt(v_hat) + adam_eps), bias-corrected).  Each of
 * `epochs` epochs draws a pseudorandom permutation pi of the S = T * n_envs samples
 * (flattened time-major, s = t * n_envs + env) and splits it into `minibatches` runs of
 * B = S / minibatches: a 4-round Feistel network on w bits (2^w >= S, w >= 2; high half
 * w - w/2 bits, low half w/2 bits; round r XORs word 0 of Philox(key = seed, counter =
 * (other half, epoch counter, 4, r)) into the high half for even r, the low half for odd
 * r), walked until the value is below S.  The epoch counter of epoch e of the k-th update
 * of a learner is k * epochs + e.
 * The network is the actor-critic ego of aht_pop_desc: obs_dim -> 128 -> 128 ->
 * n_actions + 1 (the last output is the value).  The learner keeps fp32 master weights
 * and Adam moments; the forward and backward of the update use bf16 copies of W1 and W2
 * (the precision the bf16 rollout runs) and fp32 for W3 and the biases; activations and
 * gradients are carried as two bf16 (hi + lo) through fp32-accumulating tensor cores. */
typedef struct aht_ppo_config {
  int32_t epochs;         /* >= 1 (4) */
  int32_t minibatches;    /* >= 1 (4) */
  float lr;               /* Adam step size (2.5e-4) */
  float clip_eps;         /* ratio and value clip (0.2) */
  float vf_coef;          /* value-loss weight (0.5) */
  float ent_coef;         /* entropy-bonus weight (0.01) */
  float max_grad_norm;    /* global-norm clip, <= 0 disables (0.5) */
  float adam_b1, adam_b2, adam_eps;  /* (0.9, 0.999, 1e-5) */
  uint64_t seed;          /* key of the minibatch permutations */
} aht_ppo_config;

typedef struct aht_learner aht_learner; /* opaque, library-owned */

/* Creates a PPO learner for the actor-critic ego (W[l], b[l] fp32 of the aht_pop_desc
 * shapes with hidden0 = hidden1 = 128 and the value row, host or device memory; copied).
 * obs_dim 1..207 and a multiple of 4, n_actions 1..7.  Allocates all device memory the
 * learner uses (master weights, Adam moments, the packed bf16 copy, per-SM gradient
 * partials of about 27 MB); the other learner calls allocate nothing.  Work runs on
 * cuda_stream (a cudaStream_t, NULL = default stream). */
aht_status aht_learner_create(int32_t obs_dim, int32_t n_actions, const float* const* W,
                              const float* const* b, const aht_ppo_config* cfg,
                              void* cuda_stream, aht_learner** out);
void aht_learner_destroy(aht_learner* L);
/* Number of parameters: 128 obs_dim + 128 + 128*128 + 128 + (n_actions + 1)(128 + 1). */
int64_t aht_learner_n_params(const aht_learner* L);

/* One PPO update over a trajectory of aht_rollout (device arrays obs, actions, logp,
 * values, advantages and targets of traj, [T][n_envs]; the other members are not read):
 * epochs x minibatches optimiser steps.  stats (device f32 [epochs*minibatches][6], or
 * NULL) receives per step the minibatch means of {loss, policy loss, value loss, entropy,
 * logp_old - logp, |rho - 1| > clip_eps}.  Requires T * n_envs < 2^31 and a multiple of
 * 64 * minibatches.  Asynchronous; aht_learner_sync reports device errors. */
aht_status aht_ppo_update(aht_learner* L, const aht_traj* traj, int64_t n_envs, int32_t T,
                          float* stats);
/* The gradient (device f32 [n_params], before clipping) and stats (device f32 [6], or
 * NULL) of minibatch `minibatch` of epoch `epoch` of the learner's next update, at its
 * current weights; changes nothing.  Same requirements as aht_ppo_update. */
aht_status aht_ppo_grad(aht_learner* L, const aht_traj* traj, int64_t n_envs, int32_t T,
                        int32_t epoch, int32_t minibatch, float* grad, float* stats);
/* Copies out / replaces the learner state (device f32 [n_params] arrays, each may be
 * NULL on get; params required on set, NULL moments on set mean zero): flat parameter
 * order W1, b1, W2, b2, W3, b3 (row-major), the Adam moments, step count t and the
 * number of completed updates (the permutation epoch counter is updates * epochs + e). */
aht_status aht_learner_get(aht_learner* L, float* params, float* adam_m, float* adam_v,
                           int64_t* t, int64_t* updates);
aht_status aht_learner_set(aht_learner* L, const float* params, const float* adam_m,
                           const float* adam_v, int64_t t, int64_t updates);
/* Writes the learner's current weights into policy `policy` of ctx (aht_set_policy with
 * the fp32 weights for an fp32 population, their nearest-even bf16 for a bf16 one). */
aht_status aht_learner_push(aht_learner* L, aht_ctx* ctx, int32_t policy);
/* Synchronises the learner's stream; AHT_ETIMEOUT if a bounded wait of its kernels
 * expired (the status word is then cleared). */
aht_status aht_learner_sync(aht_learner* L);

/* ---- S5 recurrent actor-critic (App. B training protocol; Sec. 4: recurrent S5 egos) ---
 * A dense relu encoder (H units, two layers), an S5 layer (Smith et al., ICLR 2023) of
 * model size H and P diagonal complex modes discretised by zero-order hold, a residual
 * GELU, and two relu MLP heads of three F-unit hidden layers (actor: n_actions logits
 * masked by the legal actions; critic: one value):
 *   u = relu(We2 relu(We1 o + be1) + be2)
 *   lbar = exp(lambda dt), Bbar = (lbar - 1) / lambda * B, dt = exp(log_dt)
 *   x_t = lbar (.) x_{t-1} + Bbar u_t  (x_{t-1} = 0 where reset),  y = Re(C x_t) + D (.) u
 *   v = u + gelu(y) (gelu(a) = a Phi(a)),  logits / value = heads(v).
 * The paper gives H = P = 128 and F = 1024; the rest is this library's reading.  Weights
 * are rounded to bf16 at create.  Hidden layers run as bf16 GEMMs (activations carried
 * as two bf16, hi + lo, ~2^-17 relative, fp32 accumulate); the SSM's products run as
 * three bf16 terms (hi hi + hi lo + lo hi, ~2^-16 relative, fp32 accumulate) and its
 * recurrence in fp32 (lbar and Bbar computed in fp64 at create); the output layers run
 * in fp32 from the fp32 last hidden layer.  Parameters are host fp32 arrays, row-major [out][in]. */
typedef struct aht_s5_params {
  int32_t obs_dim, n_actions, H, P, F;  /* obs_dim <= 2048; H, P, F multiples of 32, P <= 128;
                                           n_actions <= 32 */
  const float *We1, *be1, *We2, *be2;   /* [H][obs_dim] [H] [H][H] [H] */
  const float *lam_re, *lam_im, *log_dt;/* [P] (lam_re < 0) */
  const float *B_re, *B_im;             /* [P][H] */
  const float *C_re, *C_im;             /* [H][P] */
  const float *D;                       /* [H] */
  const float *Wa[4], *ba[4];           /* actor [F][H] [F][F] [F][F] [n_actions][F] */
  const float *Wc[4], *bc[4];           /* critic [F][H] [F][F] [F][F] [1][F] */
} aht_s5_params;
typedef struct aht_s5 aht_s5;           /* opaque, library-owned */
/* Allocates everything a step of up to max_envs envs needs (weights packed as tiled bf16
 * operands of the library's tensor-core GEMM, scratch activations).  cuda_stream: a
 * cudaStream_t (NULL = default). */
aht_status aht_s5_create(const aht_s5_params* p, int64_t max_envs, void* cuda_stream, aht_s5** out);
void aht_s5_destroy(aht_s5* s);
/* One policy step of n envs (device arrays): obs u8 [n][obs_dim], reset u8 [n] (1 zeroes
 * the env's state first: the first step of an episode), legal u8 [n][n_actions] or NULL,
 * state f32 [n][2P] in/out (real parts, then imaginary parts) -> logits f32
 * [n][n_actions] (-inf where illegal), values f32 [n].  1 <= n <= max_envs.
 * Asynchronous on the creation stream; aht_s5_sync reports errors (AHT_ETIMEOUT if a
 * product's bounded wait expired). */
aht_status aht_s5_step(aht_s5* s, const uint8_t* obs, const uint8_t* reset, const uint8_t* legal,
                       int64_t n, float* state, float* logits, float* values);
aht_status aht_s5_sync(aht_s5* s);

/* Stateless GAE (App. C "PPO ego"), time-major [T][n_envs] device arrays:
 *   delta_t = r_t + gamma (1 - d_t) V_{t+1} - V_t,
 *   A_t = delta_t + gamma lambda (1 - d_t) A_{t+1},  V_T = v_last,  A_T = 0,
 *   targets = A + V (targets may be NULL).  fp32 arithmetic; one reverse scan per env.
 * Enqueued on cuda_stream (a cudaStream_t, NULL = default). */
aht_status aht_gae(const float* rewards, const float* values, const uint8_t* dones,
                   const float* v_last, int64_t n_envs, int32_t T, float gamma, float lambda,
                   float* advantages, float* targets, void* cuda_stream);

/* Copies a collected trajectory from one set of caller-owned buffers to another: from the
 * device buffers aht_rollout wrote to pinned host buffers for a learner or a logger on
 * the host, or between device buffers (not in the paper: a transfer helper of this
 * library).  Every field that is non-NULL in both src and dst is copied in full: obs
 * [T][n_envs][obs_dim] u8, actions / tm_actions / dones [T][n_envs] u8, logp / values /
 * rewards / advantages / targets [T][n_envs] fp32, last_value [n_envs] fp32, teammate
 * [n_envs] int32; gamma and lambda are not read.  One cudaMemcpyAsync per field, in
 * this order, enqueued on cuda_stream (a cudaStream_t, NULL = default; the direction
 * follows from the pointers, and pageable host memory makes a copy synchronous); the
 * caller orders the copies after the call that wrote src (same stream, or an event).
 * AHT_EINVAL for NULL src / dst or sizes below 1, AHT_ECUDA if an enqueue fails.
 * Allocates nothing. */
aht_status aht_traj_copy(const aht_traj* src, const aht_traj* dst, int64_t n_envs, int32_t T,
                         int32_t obs_dim, void* cuda_stream);

/* Replaces the weights of one policy (App. C: PPO updates the ego between rollout
 * collections).  W[l] / b[l] (l = 0..2) have the shapes of aht_pop_desc for this policy,
 * in host or device memory of weight_dtype; has_value_head as in aht_pop_desc.  The
 * library packs them on the host into a staging buffer pinned at aht_create and
 * enqueues the upload on the context's stream; it first waits for the context's
 * previous upload.  Allocates nothing. */
aht_status aht_set_policy(aht_ctx* ctx, int32_t policy, const void* const* W,
                          const void* const* b, int32_t weight_dtype, int32_t has_value_head);

/* Kernel timing.  While enabled, the library brackets each launch of its main kernel
 * (the fused rollout of aht_rollout, the cross-play kernel of aht_xplay_matrix) with
 * CUDA events on the context's stream.  aht_get_timing synchronises the stream and
 * returns the summed kernel time in milliseconds and the number of timed launches
 * since the previous aht_get_timing (then resets both). */
aht_status aht_set_timing(aht_ctx* ctx, int32_t enable);
aht_status aht_get_timing(aht_ctx* ctx, double* kernel_ms, int64_t* launches);

/* ---- test and checkpoint hooks ------------------------------------------------ */

/* Outputs of aht_step_forced (device memory; NULL members not written). */
typedef struct aht_step_out {
  float* rewards;   /* [N][2] per-agent reward */
  float* team;      /* [N] team reward */
  uint8_t* dones;   /* [N] */
  uint8_t* obs;     /* [N][2][obs_dim] both seats' observation of the resulting state */
} aht_step_out;

/* One env step of every PPO env with the given actions (device u8 [N][2]; Hanabi uses
 * the acting seat's entry), auto-reset at step+1 as in aht_rollout, then the step
 * counter advances by 1.  An illegal Hanabi action leaves that env unchanged and
 * latches AHT_EDEVICE. */
aht_status aht_step_forced(aht_ctx* ctx, const uint8_t* actions, const aht_step_out* out);

/* Policy outputs z = MLP_p(o) for n observations: obs device u8 [n][obs_dim] ->
 * out device f32 [n][n_actions + 1] (the last column is the value row, 0 if absent). */
aht_status aht_policy_forward(aht_ctx* ctx, int32_t policy, const uint8_t* obs, int64_t n,
                              float* out);

/* The tanh of the tensor-core epilogues, elementwise: y[i] = tanh(x[i]) for device f32
 * arrays of n elements, computed for the pairs (x[2j], x[2j + 1]) as 1 - 2 / (1 + e),
 * e = exp(2x), with the hardware exp2 and reciprocal approximations and packed fp32x2
 * arithmetic; absolute error below 1e-6, tanh(0) = 0 exactly.  Stateless; enqueued on
 * cuda_stream. */
aht_status aht_debug_tanh(const float* x, float* y, int64_t n, void* cuda_stream);

/* Checkpoint of the PPO env state, the seed and the step counter into a host buffer.
 * Call with buf == NULL to get the size in *bytes.  Resuming from it is bit-exact:
 * every draw is a function of (seed, env, step, stream). */
aht_status aht_get_state(aht_ctx* ctx, void* buf, size_t* bytes);
aht_status aht_set_state(aht_ctx* ctx, const void* buf, size_t bytes);

/* Global step counter (the next step index). */
int64_t aht_step_counter(const aht_ctx* ctx);

/* Synchronises the context's stream and returns AHT_ETIMEOUT if the device status word
 * recorded only expired waits since the last aht_sync, AHT_EDEVICE if it recorded any
 * other device error (the word is then cleared), else AHT_OK. */
aht_status aht_sync(aht_ctx* ctx);

/* Failure-detection hook (no paper counterpart): enqueues on the context's stream one
 * thread that waits, with the kernels' bounded wait and a limit of limit_ns nanoseconds
 * (1 .. 10^9), on an mbarrier nothing arrives on; the wait expires and latches the
 * timeout bit, so the next aht_sync returns AHT_ETIMEOUT.  No fault, no hang. */
aht_status aht_debug_expire_wait(aht_ctx* ctx, int64_t limit_ns);

/* Allocation-failure hook (no paper counterpart), process-wide: with n >= 1 the n-th
 * device or pinned-host allocation that aht_create makes from now on fails as if the
 * device were out of memory (nothing is allocated for it), so that aht_create's unwinding
 * can be checked: it returns AHT_ENOMEM and frees everything it had allocated.  n <= 0
 * switches the hook off.  aht_debug_live_allocs returns the number of device and pinned
 * blocks that contexts hold right now (each aht_destroy returns its context's). */
aht_status aht_debug_fail_alloc(int64_t n);
int64_t aht_debug_live_allocs(void);

/* Failure-detection hook for the real kernels (no paper counterpart).  The next call of
 * aht_rollout, aht_rollout_resample, aht_rollout_ippo or aht_xplay_matrix that runs on a
 * tensor-core kernel makes its compute threads, at the call's step `step` (cross-play
 * on the streamed Overcooked / Hanabi kernel: at its launch for step `step`), wait on an
 * mbarrier nothing arrives on, in place of an accumulator wait, with the kernels' bounded
 * wait limited to limit_ns (1 .. 10^9).  The wait expires and the kernel takes its abort
 * path: it latches the timeout bit, stops, waits (bounded) for the MMAs and copies it has
 * in flight, frees its tensor memory and exits; its env state is not stored (the context
 * keeps the state from before the call; the step counter still advances by the call's
 * length) and cross-play cells of aborted tiles are NaN (LBF) or hold the returns
 * reached so far (the streamed kernel stops those envs).  The next aht_sync returns
 * AHT_ETIMEOUT.  The hook fires once; step < 0 clears it.  No fault, no hang. */
aht_status aht_debug_expire_at(aht_ctx* ctx, int32_t step, int64_t limit_ns);

/* Parity hook (no paper counterpart): the policy outputs of the tensor-core kernels,
 * element by element.  While buf (device fp32, `floats` floats, caller-owned) is set,
 * every aht_rollout, aht_rollout_resample and aht_xplay_matrix call that runs on a
 * tensor-core kernel also writes, for each policy evaluation it makes, the evaluated
 * policy's output vector (its logits, then its value row if it has one, then zeros; 8
 * entries for LBF, the padded action count for Overcooked and Hanabi) at
 * buf[((step * rows + env) * 2 + seat) * AHT_DEBUG_STRIDE ..], rows = n_envs for
 * collection and n_ego * n_tm * envs_per_pair for cross-play (whose frozen envs are
 * evaluated too); entries of seats that did not act are left as they were.  A call that
 * would write past `floats` floats returns AHT_EINVAL before it launches anything.  The
 * CUDA-core kernels do not write it.  buf == NULL turns the hook off. */
#define AHT_DEBUG_STRIDE 32
aht_status aht_debug_logits(aht_ctx* ctx, float* buf, int64_t floats);

/* Parity hook (no paper counterpart): the observation rows the streamed cross-play kernel
 * builds for Overcooked, Hanabi and Mini Hanabi contexts, for seat `seat` (0 or 1) of
 * every env's current state (Sec. 3, Omega: each agent's observation).  out: device
 * uint32 [n_envs][(obs_dim + 32) / 32], caller-owned; feature k of env e is bit k % 32 of
 * out[e][k / 32], then bit obs_dim is the constant 1 input that carries layer 1's bias,
 * and every later bit is 0.  Runs on the context's stream (aht_sync to wait).  LBF
 * contexts: AHT_EINVAL (their observations are bytes). */
aht_status aht_debug_obs_words(aht_ctx* ctx, int32_t seat, uint32_t* out);

const char* aht_last_error(void);
const char* aht_status_string(aht_status s);

#ifdef __cplusplus
}
#endif
#endif
