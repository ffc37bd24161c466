/*
 * aht_oracle.h -- plain, slow CPU oracle for the batched ad hoc teamwork rollout path.
 *
 * TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and bench.py's
 * cpu_baseline / --impl reference legs may load this library.  The product path
 * (paper_2609_13716_gb300/) never links, imports or calls it, and the two share no
 * code: no headers, helpers, tables or constants.
 *
 * What it computes (the paper is JaxAHT, "A JAX-Based Library for Ad Hoc Teamwork"):
 *   - the Dec-POMDP step of Sec. 3 (joint action -> next state, per-agent
 *     observation, one shared team reward) for three games: Level-Based Foraging,
 *     a 5x4 Overcooked-style kitchen and 2-player Hanabi (Sec. 4, Table
 *     "JaxAHT Environments").  The paper gives no game rules; the rules here are
 *     readings of the workload descriptions, stated with each game's functions below;
 *   - the decentralised MLP policy pi_i(a | o_i) (Sec. 3) in fp64 from exact weights,
 *     masked categorical sampling (App. B, masked categorical) in fp64;
 *   - PPO's generalised advantage estimate (App. C, "PPO ego") in fp64;
 *   - the ego-by-teammate cross-play return matrix (App. B, "Cross-play matrix
 *     construction"; Sec. 3 J_AHT as its row mean) and what is computed from it:
 *     best-response upper bounds, normalised returns, cooperative regret and the
 *     BRDiv cross-play objective (App. B "Upper bound estimation"; App. A);
 *   - the PPO ego update (App. C "PPO ego"): clipped-surrogate loss, its gradient, and
 *     Adam over permuted minibatches of a collected trajectory.
 * Randomness is Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11) keyed by the seed,
 * with counter (env, step, stream, block).
 *
 * All functions are re-entrant.  Array arguments are caller-owned host memory.
 */
#ifndef AHT_ORACLE_H
#define AHT_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- randomness --------------------------------------------------------------- */
enum { ORC_STREAM_ACT0 = 0, ORC_STREAM_ACT1 = 1, ORC_STREAM_RESET = 2, ORC_STREAM_TEAMMATE = 3,
       ORC_STREAM_EPISODE_TEAMMATE = 5 };

/* One Philox4x32-10 block: key (k0, k1), counter ctr[4] -> out[4]. */
void orc_philox4x32_10(uint32_t k0, uint32_t k1, const uint32_t ctr[4], uint32_t out[4]);
/* Draw n of the (env, step, stream) tuple: word n%4 of block n/4, key = (seed lo, seed hi),
 * counter = (env, step, stream, n/4). */
uint32_t orc_draw(uint64_t seed, uint32_t env, uint32_t step, uint32_t stream, uint32_t n);
/* floor(x * n / 2^32): an integer in [0, n). */
uint32_t orc_uniform_int(uint32_t x, uint32_t n);
/* (x >> 8) * 2^-24: a double in [0, 1) exactly representable in fp32. */
double orc_u01(uint32_t x);

/* ---- environment description ------------------------------------------------------ */
enum { ORC_LBF = 0, ORC_OVERCOOKED = 1, ORC_HANABI = 2, ORC_MINI_HANABI = 3 };
typedef struct orc_env_desc {
  int32_t kind;            /* ORC_LBF / ORC_OVERCOOKED / ORC_HANABI */
  int32_t width, height;   /* LBF grid (3..12); Overcooked 5x4; Hanabi ignored */
  int32_t n_food;          /* LBF 1..3 */
  int32_t max_agent_level; /* LBF agent levels are uniform in 1..max_agent_level */
  int32_t episode_len;     /* LBF / Overcooked step limit; Hanabi 0 = run to termination */
  int32_t cook_time;       /* Overcooked steps a full pot cooks */
  int32_t soup_reward;     /* Overcooked team reward per delivered soup */
} orc_env_desc;

int32_t orc_obs_dim(const orc_env_desc* d);
int32_t orc_n_actions(const orc_env_desc* d);
/* 0 if the description is valid, else a negative code. */
int32_t orc_check_desc(const orc_env_desc* d);

/* ---- Level-Based Foraging -------------------------------------------------------- */
enum { ORC_LBF_MAX_FOOD = 3 };
typedef struct orc_lbf_state {
  int32_t ax[2], ay[2], al[2];         /* agent position and level */
  int32_t fx[3], fy[3], fl[3], eaten[3];
  int32_t F;                           /* sum of spawned food levels (reward normaliser) */
  int32_t ep_t;                        /* steps taken in this episode */
  int32_t done;                        /* the last step ended the episode */
  float ret;                           /* team return of this episode */
  int32_t ix[2], iy[2];                /* agent positions at the episode's start */
} orc_lbf_state;
void orc_lbf_reset(const orc_env_desc* d, uint64_t seed, uint32_t env, uint32_t step,
                   orc_lbf_state* s);
/* r[2] = per-agent reward, *team = fp32(r0 + r1).  Returns done (0/1). */
int32_t orc_lbf_step(const orc_env_desc* d, orc_lbf_state* s, int32_t a0, int32_t a1,
                     float r[2], float* team);
void orc_lbf_obs(const orc_env_desc* d, const orc_lbf_state* s, int32_t seat, uint8_t* out);

/* Rule-based LBF teammates (App. F, LBF heuristic suite: Greedy picks the next uneaten
 * food online by a criterion, Sequential plans a food order before the episode).  The
 * paper names the criteria and orderings only; the rules are these readings:
 *   k = 0..4  Greedy: argmin over uneaten foods of dist(self) | dist(teammate) |
 *             dist(self) + dist(teammate) | level | -level (ties: lower food index);
 *   k = 5..10 Sequential: the first uneaten food in the order of row-major cell index
 *             (y W + x) ascending | descending, column-major index (x H + y) ascending |
 *             descending, distance from the agent's position at the episode's start
 *             ascending | descending (ties: lower food index);
 * then the action toward it: load (5) when 4-adjacent; else a step along the axis with
 * the larger remaining distance (ties: x), or along the other axis if that cell is off
 * the grid, an uneaten food or the other agent; else noop.  dist is Manhattan.
 *   k = 11    Entitled: for the lowest-index uneaten food, the pair of squares is its
 *             first two 4-neighbours in the order W, E, N, S that are on the grid and
 *             hold no uneaten food (fewer than two: noop); while the other
 *             agent stands on neither, noop; once it stands on one, go to the other (the
 *             step rule above, toward that cell) and load when standing on it.
 * A teammate id t < 0 in a pool or teammate list means heuristic k = -1 - t (LBF only). */
enum { ORC_LBF_N_HEURISTICS = 12 };
int32_t orc_lbf_heuristic(const orc_env_desc* d, const orc_lbf_state* s, int32_t seat, int32_t k);

/* ---- Overcooked-style kitchen (fixed 5x4 layout) -------------------------------- */
enum { ORC_OC_NONE = 0, ORC_OC_ONION = 1, ORC_OC_DISH = 2, ORC_OC_SOUP = 3 };
enum { ORC_OC_FLOOR = 0, ORC_OC_COUNTER = 1, ORC_OC_ONION_D = 2, ORC_OC_POT = 3,
       ORC_OC_DISH_D = 4, ORC_OC_SERVE = 5 };
typedef struct orc_oc_state {
  int32_t ax[2], ay[2], face[2], held[2]; /* face 0 N, 1 S, 2 E, 3 W */
  int32_t pot_n, pot_timer;
  int32_t counter_item[20];               /* item on each cell (counters only) */
  int32_t ep_t;
  int32_t done;
  float ret;
} orc_oc_state;
int32_t orc_oc_cell(int32_t x, int32_t y); /* layout cell type */
void orc_oc_reset(const orc_env_desc* d, orc_oc_state* s);
int32_t orc_oc_step(const orc_env_desc* d, orc_oc_state* s, int32_t a0, int32_t a1,
                    float r[2], float* team);
void orc_oc_obs(const orc_env_desc* d, const orc_oc_state* s, int32_t seat, uint8_t* out);

/* ---- Hanabi, 2 players ------------------------------------------------------------ */
typedef struct orc_hanabi_state {
  int32_t deck[50];           /* card type c*5 + (rank-1) */
  int32_t ptr;                /* next card to draw */
  int32_t hand[2][5];         /* card type, -1 if empty */
  int32_t n_hand[2];
  uint32_t know[2][5];        /* 25-bit possible-card masks */
  uint32_t hint_col[2][5];    /* explicit colour hints received, 5 bits */
  uint32_t hint_rank[2][5];   /* explicit rank hints received, 5 bits */
  int32_t fw[5];              /* fireworks height per colour */
  int32_t info, lives, score;
  int32_t disc[25];           /* discarded count per card type */
  int32_t fr;                 /* final-round turns left; -1 while the deck has cards */
  int32_t turn;               /* turns taken in this episode; acting seat = turn % 2 */
  int32_t la_valid, la_actor, la_type, la_colour, la_rank, la_slot, la_card, la_hinted,
          la_success, la_bomb; /* last action */
  int32_t done;
  float ret;
} orc_hanabi_state;
void orc_hanabi_reset(uint64_t seed, uint32_t env, uint32_t step, orc_hanabi_state* s);
void orc_hanabi_legal(const orc_hanabi_state* s, uint8_t legal[20]); /* for the acting seat */
/* Applies action a of the acting seat.  Returns done (0/1), or -1 (state untouched)
 * if a is illegal. */
int32_t orc_hanabi_step(orc_hanabi_state* s, int32_t a, float* team);
void orc_hanabi_obs(const orc_hanabi_state* s, int32_t seat, uint8_t* out);

/* ---- Mini Hanabi, 2 players (Sec. 4 Table "JaxAHT Environments": 3 colours x 3 ranks).
 * The paper gives only the colour and rank counts; the rest is this reading:
 * 18-card deck (ranks 1,1,1,2,2,3 per colour), 2-card hands, 3 info and 1 life tokens,
 * 10 actions (play slot 0-1, discard slot 0-1, hint colour 0-2, hint rank 1-3), card type
 * = colour*3 + rank-1, and the full game's rules and observation sections at this size
 * (153 bits, then 3 zero features: 156).  The library stops any game at 100 turns. */
typedef struct orc_mhanabi_state {
  int32_t deck[18];
  int32_t ptr;
  int32_t hand[2][2];         /* card type, -1 if empty */
  int32_t n_hand[2];
  uint32_t know[2][2];        /* 9-bit possible-card masks */
  uint32_t hint_col[2][2];    /* 3 bits */
  uint32_t hint_rank[2][2];   /* 3 bits */
  int32_t fw[3];
  int32_t info, lives, score;
  int32_t disc[9];
  int32_t fr;
  int32_t turn;
  int32_t la_valid, la_actor, la_type, la_colour, la_rank, la_slot, la_card, la_hinted,
          la_success, la_bomb;
  int32_t done;
  float ret;
} orc_mhanabi_state;
void orc_mhanabi_reset(uint64_t seed, uint32_t env, uint32_t step, orc_mhanabi_state* s);
void orc_mhanabi_legal(const orc_mhanabi_state* s, uint8_t legal[10]);
int32_t orc_mhanabi_step(orc_mhanabi_state* s, int32_t a, float* team);
void orc_mhanabi_obs(const orc_mhanabi_state* s, int32_t seat, uint8_t* out);

/* ---- generic env state ------------------------------------------------------------ */
enum { ORC_STATE_BYTES = 768 };   /* >= sizeof of every state struct above */
typedef struct orc_state { uint8_t bytes[ORC_STATE_BYTES]; } orc_state;

/* ---- policy MLP ------------------------------------------------------------------ */
typedef struct orc_mlp {
  int32_t obs_dim, h0, h1, n_out; /* n_out = n_actions, + 1 if a value row is present */
  const double *W1, *b1;          /* [h0][obs_dim], [h0] */
  const double *W2, *b2;          /* [h1][h0], [h1] */
  const double *W3, *b3;          /* [n_out][h1], [n_out] */
} orc_mlp;
/* z = W3 tanh(W2 tanh(W1 x + b1) + b2) + b3, fp64. */
void orc_mlp_forward(const orc_mlp* p, const double* x, double* z);
/* Masked categorical inverse-CDF sample in fp64: a = min{k : u*Z < S_k}, with
 * S_k = sum_{j<=k} exp(z_j - max) over legal j.  logp of a; margin = min_k |u - S_k/Z|. */
void orc_sample(const double* z, const uint8_t* legal, int32_t K, double u,
                int32_t* a, double* logp, double* margin);
/* logp of a given action under the masked softmax of z. */
double orc_logp(const double* z, const uint8_t* legal, int32_t K, int32_t a);

/* ---- GAE (fp64) -------------------------------------------------------------------- */
/* Time-major [T][N] inputs.  delta_t = r_t + g(1-d_t)V_{t+1} - V_t,
 * A_t = delta_t + g l (1-d_t) A_{t+1}, V_T = v_last, A_T = 0; targets = A + V. */
void orc_gae(const float* r, const float* v, const uint8_t* d, const float* v_last,
             int64_t n_envs, int32_t T, double gamma, double lambda,
             double* adv, double* targets);

/* ---- PPO rollout collection (simultaneous-move envs) ---------------------------- */
/* Teammates (Sec. 3: the ego meets teammates drawn from the training set).  Per-call
 * mode: every env draws its own teammate once per call, at the call's first step --
 * env e plays pool[uniform_int(x, pool_size)], x = word 0 of counter (e, step0,
 * stream 3) -- and keeps it for the whole call, auto-reset episodes included.
 * Per-episode mode (resample = 1): each episode draws its own teammate when it begins --
 * env e whose current episode began at step s plays pool[uniform_int(x, pool_size)],
 * x = word 0 of counter (e, s, stream 5); the step an episode began is carried per env
 * in ep_step (0 after a reset of the whole batch), and every auto-reset at step s' sets
 * it to s'. */
typedef struct orc_rollout_io {
  /* inputs */
  uint64_t seed;
  int64_t n_envs;
  int64_t step0;               /* global step counter at the start of the call */
  int32_t T;
  int32_t ego_id;
  const int32_t* pool;         /* teammate policy ids */
  int32_t pool_size;
  const uint8_t* forced;       /* [T][N][2] actions to apply, or NULL to free-run */
  const int64_t* env_ids;      /* [N] global env index of each row, or NULL for 0..N-1 */
  orc_state* states;           /* [N] in/out */
  int32_t n_threads;
  /* outputs (each may be NULL) */
  int32_t* teammate;           /* [N] */
  uint8_t* obs;                /* [T][N][obs_dim] ego observation */
  uint8_t* obs_tm;             /* [T][N][obs_dim] teammate observation */
  uint8_t* actions;            /* [T][N][2] applied actions */
  uint8_t* own_actions;        /* [T][N][2] the oracle's own samples */
  double* margin;              /* [T][N][2] CDF margin of each own sample */
  double* logits;              /* [T][N][n_out] ego outputs */
  double* logp;                /* [T][N] ego logp of the applied action */
  double* values;              /* [T][N] ego value (0 without a value row) */
  float* rewards;              /* [T][N] team reward */
  uint8_t* dones;              /* [T][N] */
  double* last_value;          /* [N] value of the state after the last step */
  /* the teammate seat's learner outputs (IPPO, both seats learn; 0 for a rule teammate) */
  double* logp_tm;             /* [T][N] teammate logp of its applied action */
  double* values_tm;           /* [T][N] teammate value (0 without a value row) */
  double* last_value_tm;       /* [N] teammate value of the state after the last step */
  /* per-episode teammates */
  int32_t resample;            /* 0: per-call mode, 1: per-episode mode (ep_step required) */
  uint32_t* ep_step;           /* [N] in/out, or NULL in per-call mode */
  int32_t* teammates_t;        /* [T][N] teammate policy id at each step, or NULL */
} orc_rollout_io;
int32_t orc_rollout(const orc_env_desc* d, const orc_mlp* pols, int32_t n_pols,
                    orc_rollout_io* io);

/* Resets n_envs envs with env index 0..n-1 at the given step counter. */
int32_t orc_reset_all(const orc_env_desc* d, uint64_t seed, int64_t n_envs, int64_t step,
                      orc_state* states);
/* Resets the envs with the given global indices (row i gets env ids[i]). */
int32_t orc_reset_envs(const orc_env_desc* d, uint64_t seed, const int64_t* ids, int64_t n,
                       int64_t step, orc_state* states);
/* One forced step of every env, PPO semantics (auto-reset with step+1).  Outputs the
 * per-agent rewards [N][2], team rewards [N], dones [N] and both seats' observation of
 * the resulting state [N][2][obs_dim]; each output may be NULL.  Hanabi applies the
 * acting seat's action only. */
int32_t orc_step_forced(const orc_env_desc* d, uint64_t seed, int64_t n_envs, int64_t step,
                        orc_state* states, const uint8_t* actions, float* rewards2,
                        float* team, uint8_t* dones, uint8_t* obs2);

/* ---- cross-play evaluation ------------------------------------------------------- */
typedef struct orc_xplay_io {
  uint64_t seed;
  int64_t step0;
  const int32_t* ego_ids; int32_t n_ego;
  const int32_t* tm_ids;  int32_t n_tm;
  int32_t envs_per_pair;
  int32_t max_steps;
  const uint8_t* forced;   /* [max_steps][n_envs][2] or NULL */
  const int64_t* env_ids;  /* [n_sel] global env indices to run, or NULL for all envs;
                              outputs are then indexed by selection row */
  int64_t n_sel;
  int32_t n_threads;
  /* outputs (each may be NULL) */
  float* returns;          /* [n_ego][n_tm][P] team return of the first episode */
  int32_t* steps;          /* [n_envs] active env-steps */
  uint8_t* actions;        /* [max_steps][n_envs][2] applied actions (255 = none) */
  uint8_t* own_actions;    /* [max_steps][n_envs][2] */
  double* margin;          /* [max_steps][n_envs][2] (2 = no sample) */
  float* matrix;           /* [n_ego][n_tm] mean return, fp64 sum (all envs only) */
  double* logits;          /* [max_steps][n_envs][2][logit_stride]: the acting seats'
                              policy outputs (untouched where a seat did not act) */
  int32_t logit_stride;
} orc_xplay_io;
int32_t orc_xplay(const orc_env_desc* d, const orc_mlp* pols, int32_t n_pols,
                  orc_xplay_io* io);

/* ---- Cross-play matrix consumers (fp64) ------------------------------------------ */
/* xp [n_ego][n_tm]: rows are the policies in the ego seat (best responses, or the ego),
 * columns the evaluation teammates.
 *   upper[m] (in/out), App. B "Upper bound estimation": the recorded bound of teammate m
 *     is replaced by each XP score of column m that exceeds it, rows in order (strict >,
 *     so a NaN bound stays NaN; pass -inf for "no bound yet").
 *   norm[e][m] = xp[e][m] / upper[m], the return relative to the best response's
 *     (Sec. 3; App. B "normalized return"); NaN where upper[m] <= 0.
 *   regret[e][m] = upper[m] - xp[e][m], the cooperative regret of App. A (ROTATE):
 *     best-response return minus the return of the row's policy.
 *   j_aht[e] = (1/n_tm) sum_m xp[e][m], Sec. 3 J_AHT with T_eval uniform; j_norm[e] the
 *     same mean of norm[e][.] (unrounded fp64 terms).
 *   max_regret[e] = max_m regret[e][m] (strict >, lowest m wins ties), worst[e] that m.
 *   brdiv (n_ego == n_tm only; NULL otherwise) = (1/n) sum_i xp[i][i]
 *     - (1/(n(n-1))) sum_i sum_{j != i} xp[i][j]: matched teammate/best-response returns
 *     up, mismatched cross-play down (App. A, BRDiv), unit weights; the second term is 0
 *     for n = 1.
 * Every sum runs left to right in fp64; the off-diagonal sum adds each row's own partial
 * sum, rows in order.  Output pointers other than upper may be NULL. */
void orc_xp_stats(const float* xp, int32_t n_ego, int32_t n_tm, double* upper, double* norm,
                  double* regret, double* j_aht, double* j_norm, double* max_regret,
                  int32_t* worst, double* brdiv);

/* ---- PPO ego update (fp64; ppo_oracle.cpp) -------------------------------------- */
/* App. C "PPO ego": PPO (Schulman et al. 2017) with the clipped surrogate, a clipped
 * value loss and an entropy bonus, per-minibatch advantage normalisation, global-norm
 * gradient clipping and Adam (Kingma & Ba 2015); the paper states neither the loss nor
 * the hyperparameters, so the settings are those orc_ppo_hp carries (defaults: 4 epochs x
 * 4 minibatches, clip 0.2, value 0.5, entropy 0.01, gradient norm 0.5, Adam 0.9 / 0.999 /
 * 1e-5, lr 2.5e-4).
 * Parameters are one flat array: W1 [h0][obs_dim], b1 [h0], W2 [h1][h0], b2 [h1],
 * W3 [n_act + 1][h1], b3 [n_act + 1] (the last output row is the value estimate). */
enum { ORC_STREAM_PERMUTE = 4 };
typedef struct orc_ppo_net {
  int32_t obs_dim, h0, h1, n_act;
} orc_ppo_net;
typedef struct orc_ppo_hp {
  int32_t epochs, minibatches;
  double lr, clip_eps, vf_coef, ent_coef, max_grad_norm, adam_b1, adam_b2, adam_eps;
  uint64_t seed;      /* minibatch permutation key */
  int64_t epoch0;     /* permutation counter of the first epoch */
  int32_t round_bf16; /* 1: the forward and backward use bf16(W1), bf16(W2) */
} orc_ppo_hp;
/* Samples s in [0, S): the [T][N] trajectory arrays flattened time-major (s = t*N + n). */
typedef struct orc_ppo_batch {
  const uint8_t* obs;       /* [S][obs_dim] */
  const uint8_t* actions;   /* [S] */
  const float* logp;        /* [S] log-probability under the rollout policy */
  const float* values;      /* [S] value estimate of the rollout */
  const float* advantages;  /* [S] GAE */
  const float* targets;     /* [S] value targets (advantages + values) */
} orc_ppo_batch;
int64_t orc_ppo_n_params(const orc_ppo_net* n);
/* bf16 nearest-even of fp32(w). */
double orc_bf16_round(double w);
/* pi_epoch(x) for x in [0, S): a 4-round Feistel network on the smallest w >= 2 bits
 * with 2^w >= S (high half L = w - w/2 bits, low half R = w/2 bits; round r XORs the low
 * half's Philox word into L for even r, the high half's into R for odd r, Philox key
 * (seed lo, seed hi), counter (other half, epoch, ORC_STREAM_PERMUTE, r), word 0), walked
 * until the value falls below S.  Minibatch b of epoch e is pi_e(b*B .. (b+1)*B - 1). */
int64_t orc_perm_index(uint64_t seed, int64_t epoch, int64_t S, int64_t x);
/* Gradient of the minibatch loss at params over the B samples idx[] (the loss is the
 * mean over them); stats (may be NULL) = {loss, policy loss, value loss, entropy,
 * mean(logp_old - logp), fraction with |ratio - 1| > clip_eps}. */
void orc_ppo_grad(const orc_ppo_net* n, const double* params, const orc_ppo_batch* tb,
                  const int64_t* idx, int64_t B, const orc_ppo_hp* hp, double* grad,
                  double* stats, int32_t n_threads);
/* One optimiser step: clip grad (in place) to global norm max_grad_norm (if > 0), t += 1,
 * Adam with bias correction, params -= lr m_hat / (sqrt(v_hat) + adam_eps). */
void orc_adam_step(int64_t n_params, double* params, double* m, double* v, int64_t* t,
                   double* grad, const orc_ppo_hp* hp);
/* epochs x minibatches steps over S samples (B = S / minibatches); stats [E*M][6]. */
void orc_ppo_update(const orc_ppo_net* n, double* params, double* m, double* v, int64_t* t,
                    const orc_ppo_batch* tb, int64_t S, const orc_ppo_hp* hp, double* stats,
                    int32_t n_threads);

/* Policy outputs z for n observations (u8 [n][obs_dim]) -> [n][n_out]. */
void orc_policy_outputs(const orc_mlp* p, const uint8_t* obs, int64_t n, double* out);

/* ---- S5 recurrent actor-critic (App. B "Training protocol", Sec. 4: recurrent S5 ego
 * agents) ------------------------------------------------------------------------------
 * The paper: observations go through dense layers into an S5 sequence model of model
 * size H = 128 and SSM state size P = 128 (Smith, Warrington, Linderman, "Simplified State
 * Space Layers for Sequence Modeling", ICLR 2023), then separate MLP heads with three
 * hidden layers of 1024 units give a masked categorical policy and a value.  Readings
 * (the rest is unstated):
 *   encoder u = relu(We2 relu(We1 o + be1) + be2)   (o the u8 observation, E = H units)
 *   SSM, P diagonal complex modes, zero-order hold with step dt_p = exp(log_dt_p):
 *     lbar_p = exp(lambda_p dt_p),  Bbar[p][:] = (lbar_p - 1) / lambda_p * B[p][:]
 *     x_t = lbar (.) x_{t-1} + Bbar u_t  (x_{t-1} = 0 at an episode's first step)
 *     y_t = Re(C x_t) + D (.) u_t          (B: P x H complex, C: H x P complex, D: H real)
 *   v_t = u_t + gelu(y_t),  gelu(a) = a Phi(a) (the exact form, Phi the normal CDF)
 *   heads: relu MLPs H -> F -> F -> F -> n_actions (actor) and -> 1 (critic), F = 1024;
 *   the actor's logits are masked by the legal actions when given.
 * The state is carried per env as 2P doubles (real parts, then imaginary parts). */
typedef struct orc_s5_net {
  int32_t obs_dim, n_actions, H, P, F;
  const double *We1, *be1, *We2, *be2;       /* [H][obs_dim] [H] [H][H] [H] */
  const double *lam_re, *lam_im, *log_dt;    /* [P] each, lam_re < 0 */
  const double *B_re, *B_im;                 /* [P][H] */
  const double *C_re, *C_im;                 /* [H][P] */
  const double *Dv;                          /* [H] */
  const double *Wa[4], *ba[4];               /* actor [F][H] [F][F] [F][F] [A][F], biases */
  const double *Wc[4], *bc[4];               /* critic [F][H] [F][F] [F][F] [1][F], biases */
} orc_s5_net;
/* u = encoder(o) [H]. */
void orc_s5_encode(const orc_s5_net* n, const uint8_t* obs, double* u);
/* One SSM step: state [2P] in/out (zeroed first when reset), y [H]. */
void orc_s5_ssm_step(const orc_s5_net* n, const double* u, int32_t reset, double* state, double* y);
/* Heads on v [H]: logits [n_actions] (-inf where legal[a] == 0, legal may be NULL), value. */
void orc_s5_heads(const orc_s5_net* n, const double* v, const uint8_t* legal, double* logits,
                  double* value);
/* One full step for n envs: obs u8 [n][obs_dim], reset [n], legal u8 [n][A] or NULL,
 * state [n][2P] in/out -> logits [n][A], values [n]. */
void orc_s5_step(const orc_s5_net* net, const uint8_t* obs, const uint8_t* reset,
                 const uint8_t* legal, int64_t n, double* state, double* logits, double* values,
                 int32_t n_threads);

#ifdef __cplusplus
}
#endif
#endif
