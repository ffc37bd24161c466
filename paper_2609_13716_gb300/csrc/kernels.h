// kernels.h -- launch interface between the C-ABI layer (aht_api.cu) and the kernels.
#pragma once
#include "aht_common.cuh"

namespace aht {

struct TrajPtrs {
  uint8_t* obs;
  uint8_t* actions;
  uint8_t* tm_actions;
  float* logp;
  float* values;
  float* rewards;
  uint8_t* dones;
  float* last_value;
};

// Common per-launch description of the env batch and the population.
struct Batch {
  DevEnv env;
  MlpDims mlp;
  const float* weights;  // packed population
  Key key;
  uint32_t* status;      // device status word
};

struct PpoArgs {
  Batch b;
  uint32_t* state;       // SoA env state [kWords][n_envs]
  int64_t n_envs;
  const int32_t* perm;   // env ids grouped by teammate
  const int4* tiles;     // (perm offset, count, teammate policy, -)
  int32_t M;             // rows per tile
  int32_t ego;
  uint32_t step0;
  int32_t T;
  uint32_t* ep_step;     // [n_envs] step each env's episode began, set at every auto-reset
  TrajPtrs traj;
  TrajPtrs traj1;        // seat 1's learner trajectory (IPPO); all NULL otherwise: obs,
                         // actions = its own, tm_actions = seat 0's, logp, values,
                         // rewards, dones, last_value of the seat-1 policy
};

// Per-policy block of the tensor-core path (byte offsets within the block):
//   W1 [H0][KP] bf16, canonical K-major (see tc_common.cuh); column obs_dim holds b1
//      (the observation tile carries a constant 1 there),
//   W2 [H1][H0] bf16, canonical K-major,
//   W3 [H1 * 32 bytes]: bf16 B fragments of mma.sync m16n8k16, [H1 / 16 unit chunks j]
//      [32 threads t][2 words], word i of thread t holding W3[t / 4][16 j + 8 i + 2 (t % 4)]
//      in its low and W3[t / 4][... + 1] in its high half (outputs past n_actions, and the
//      value row when absent, are zero); split blocks follow with the bf16 remainders
//      W3 - bf16(W3) in the same layout at + H1 * 16 bytes,
//   b2 fp32 [H1], b3 fp32 [8],
// where the layers above a hidden layer hold the affine map of its logistic activation
// r = 1 / (1 + exp(2x)) = (1 - tanh(x)) / 2 (the kernels' activation): W2 and W3 are
// stored as -2 W (exact), b3 as b3 + W3 1 and b2 as (b2 + W2 1) 2 / ln 2 (the scale of
// epilogue 2's exponent; sums in fp64, rounded once),
// and for fp32 populations ("split" blocks) W1lo and W2lo, the bf16 remainders
// W - bf16(W) in the same layouts as W1 and W2: W = W1 + W1lo to about 2^-17 relative
// (the weight of the constant-1 input likewise carries b1 as two parts).
struct TcDims {
  int32_t KP, H0, H1;      // padded obs dim (> obs_dim), hidden sizes
  int32_t split;           // 1: fp32 weights as bf16 pairs (W1lo, W2lo present)
  int32_t sparse;          // 1: no W1 in the block; the first layer runs on CUDA cores from
                           // the env's changed features and the fp32 W1^T / c of the
                           // CUDA-core population (LBF grids beyond 256 tensor-memory columns)
  uint32_t oW1, oW2, oW3, ob2, ob3, oW1lo, oW2lo;
  uint32_t pol_bytes;
};

// Cross-play tiles of the tensor-core rollout kernel: tile t is chunk t % tpp of pair
// t / tpp, envs [pair P + 128 chunk, min(pair P + 128 chunk + 128, (pair + 1) P)), ego
// ego_ids[pair / n_tm], teammate tm_ids[pair % n_tm].
struct TcXp {
  int32_t n_tm, P, tpp, max_steps;
  int64_t n_total;
  int32_t ego_ids[kMaxXpIds];
  int32_t tm_ids[kMaxXpIds];
  float* returns;          // [n_total]
  int32_t* steps;          // optional [n_total]
  uint8_t* actions;        // optional [max_steps][n_total][2], pre-filled with 255
};

// Gathered tiles of the tensor-core rollout: the envs of one tile share a teammate's
// pool index but are not a contiguous range.  Each env carries its pool index (kidx) and
// the launch the envs per index (hist).  CTA j takes tile j of the groups laid out in
// pool-index order (each group cut into tiles of up to M envs in env order) and finds
// its envs by a rank scan of kidx.
//   Per call (resample = 0): kidx / hist of the call's draw; the tile keeps its envs for
//   all T steps of the launch.
//   Per episode (resample = 1, one launch per step): kidx double-buffered and hist
//   triple-buffered by step; the launch writes each env's index for the next step (a new
//   draw after an auto-reset) and adds the next step's counts; CTA 0 zeroes the buffer
//   the step after next will count into.
struct TcGather {
  const uint8_t* kidx_cur;  // [N] pool index per env at this step (16-byte aligned)
  uint8_t* kidx_next;       // [N] at the next step (per episode)
  const int32_t* hist_cur;  // [pool_size] envs per index at this step
  int32_t* hist_next;       // [pool_size] accumulated for the next step (per episode; zero on entry)
  int32_t* hist_zero;       // [pool_size] zeroed by CTA 0 (per episode)
  int32_t* teammate;        // optional [N]: policy of each env at this step (per episode)
  int32_t* teammate2;       // optional second copy (per episode)
  uint32_t scratch_off;     // dynamic shared-memory offset of the scan scratch
  int32_t resample;         // 1: per-episode mode
  int32_t M;                // rows per tile (32, 64 or 128)
  int32_t pool_size;
  int32_t pool[kMaxPool];
};
constexpr uint32_t kTcGatherScratch = 128 * 4 + 32 * 4;  // row envs, warp totals, selection

struct PpoTcArgs {
  Batch b;
  TcDims tc;
  const uint8_t* tcw;    // [n_policies][pol_bytes]
  uint32_t* state;
  int64_t n_envs;
  const int4* tiles;     // tiles of up to 128 contiguous envs (not read by gather launches)
  int32_t ego;
  uint32_t step0;
  int32_t T;
  uint32_t* ep_step;     // as in PpoArgs
  int32_t gather;        // gathered tiles (see TcGather)
  TrajPtrs traj;
  TrajPtrs traj1;        // as in PpoArgs
  TcXp xp;               // cross-play launches only
  TcGather g;            // gather launches only
  float* dbg_logits;     // test hook, or NULL: [steps][rows][2 seats][kDbgStride] outputs
  int32_t dbg_expire_step;   // test hook: at this step the compute threads wait, bounded by
  uint64_t dbg_expire_ns;    // dbg_expire_ns, on an mbarrier nothing arrives on (-1: never)
  int32_t pdl;               // launch as a programmatic dependent of the stream's previous
                             // kernel (the two-group kernel only; its setup overlaps that kernel)
};

// Per-policy block of the streamed tensor-core path (binary observations, hidden width H
// = 256 or 512 for both layers).  W1 and W2 are cut into 8 KB chunks, each a [256][16]
// bf16 slice (256 output rows, 16 inputs) in the canonical K-major layout, so that one
// chunk is the B operand of one N = 256, K = 16 MMA:
//   chunk nh * (KP / 16) + ks            W1 rows [256 nh, 256 nh + 256), inputs [16 ks, 16 ks + 16)
//   n_l1 + nh * (H / 16) + ks            W2 likewise (inputs are layer-1 units)
// Input column obs_dim of W1 holds b1 (the observation carries a constant 1 there).
// Then W3 as bf16 B fragments of mma.sync m16n8k16 (the output layer runs on the legacy
// tensor-core path from registers): [H / 16 unit chunks j][ceil(NAP / 8) n-tiles][32
// threads t][2 words], word i of thread t holding W3[8 nt + t / 4][16 j + 8 i + 2 (t % 4)]
// in its low and W3[same][... + 1] in its high half (zero past the outputs); b2 fp32 [H],
// b3 fp32 [NAP].
struct WideDims {
  int32_t KP, H, NAP;      // padded input (a multiple of 16), hidden width, padded outputs
  int32_t n_l1, n_l2;      // chunks of W1 and W2
  uint32_t oW3, ob2, ob3;  // byte offsets
  uint32_t pol_bytes;
};
constexpr uint32_t kWideChunk = 8192;

// One launch = one step s of a cross-play batch (see xplay_tc.cuh).
struct XpTcArgs {
  Batch b;
  WideDims w;
  const uint8_t* tcw;      // [n_policies][pol_bytes]
  int32_t n_ego, n_tm, P, max_steps, s;
  int32_t ego_ids[kMaxXpIds];
  int32_t tm_ids[kMaxXpIds];
  uint32_t step0;
  int64_t n_total;         // n_ego * n_tm * P
  const uint32_t* st_in;   // SoA state [words][n_total]: after step s - 1
  uint32_t* st_out;        // after step s (written by the owning tiles)
  int32_t parts;           // CTAs per tile: 2 split layer 2 by N = 256 block (H = 512), else 1
  const uint8_t* act_in;   // one part: [n_total][2] actions of step s - 1
  uint8_t* act_out;        // one part: [n_total][2] actions of step s
  const float* zp_in;      // two parts: [n_total][2 seats][2 parts][NAP] outputs of step s - 1,
  float* zp_out;           //   without b3; those of step s (each part writes its slot)
  const uint8_t* alive_in; // [n_total]
  uint8_t* alive_out;
  int32_t* nsteps;         // [n_total] steps taken
  float* returns;          // [n_total]
  int32_t* steps;          // optional [n_total]
  uint8_t* actions;        // optional [max_steps][n_total][2]
  float* dbg_logits;       // test hook, or NULL: [max_steps][n_total][2 seats][kDbgStride]
  int32_t dbg_expire_step; // test hook: launch s == this waits on an mbarrier nothing
  uint64_t dbg_expire_ns;  // arrives on, bounded by dbg_expire_ns (-1: never)
  // Two parts (H = 512): each computes one N = 256 block of L1 and the parts swap their
  // hidden units' bf16 halves through L2-resident memory: CTA b's slot of kXchSlot bytes
  // at xch + b kXchSlot, published by xflag[b] = 2 xstamp (2 xstamp + 1: the CTA gave up).
  // xstamp is unique per launch of a context, so no flag needs clearing between launches.
  uint8_t* xch;
  uint32_t* xflag;
  uint32_t xstamp;
};
// One part's exchange slot: hi and lo of 256 hidden units x 128 rows, bf16, as 16-byte
// chunks of 8 units, [hi 32 | lo 32 chunks][128 rows].
constexpr size_t kXchSlot = 2 * 32 * 128 * 16;

// Test hook layout: every policy evaluation of a tensor-core kernel may write its output
// vector (logits, then the value where the policy has one, then zeros) at
// [step][row][seat][0 .. kDbgStride).
constexpr int kDbgStride = 32;

// Teammate assignment of one collection call (per-call draw, counter (e, step0, stream 3)).
struct GroupArgs {
  Key key;
  int64_t n_envs;
  uint32_t step0;
  int32_t pool_size;
  int32_t pool[kMaxPool];
  int32_t M;
  int32_t max_tiles;
  int32_t* perm;         // group_kernel (one-member pool): identity
  int4* tiles;           // group_kernel: contiguous tiles of up to M envs
  int32_t* teammate;     // optional [n_envs]
  uint8_t* kidx;         // teammate_draw_kernel: [n_envs] pool index per env
  int32_t* hist;         // teammate_draw_kernel: [pool_size] += envs per index (zeroed before)
};

// Teammates grouped for the CUDA-core rollout: env e plays pool[uniform_int(x, pool_size)]
// with x the first draw of counter (e, ep_step[e], stream 5) per episode, or of (e, step0,
// stream 3) per call when ep_step is NULL; perm lists the envs grouped by pool index,
// tiles (perm offset, count, policy, -) cover each group in tiles of up to M envs.
struct ResampleGroupArgs {
  Key key;
  int64_t n_envs;
  uint32_t step0;
  const uint32_t* ep_step;
  int32_t pool_size;
  int32_t pool[kMaxPool];
  int32_t M;
  int32_t max_tiles;
  int32_t* perm;
  int4* tiles;
  int32_t* teammate;     // optional [n_envs]: the policy each env plays at this step
  int32_t* teammate2;    // optional second copy (the call's first step)
};

struct XpArgs {
  Batch b;
  int32_t n_ego, n_tm, P, max_steps;
  int32_t ego_ids[kMaxXpIds];
  int32_t tm_ids[kMaxXpIds];
  int32_t M, tiles_per_pair;
  uint32_t step0;
  float* returns;        // [n_pairs * P]
  int32_t* steps;        // optional
  uint8_t* actions;      // optional [max_steps][n][2]
};

struct ForcedArgs {
  Batch b;
  uint32_t* state;
  int64_t n_envs;
  uint32_t step;
  const uint8_t* actions;  // [N][2]
  float* rewards;          // [N][2]
  float* team;
  uint8_t* dones;
  uint8_t* obs;            // [N][2][obs_dim]
  uint32_t* ep_step;       // optional [N]
};

struct ResetArgs {
  Batch b;
  uint32_t* state;
  int64_t n_envs;
  uint32_t step;
  uint32_t* ep_step;       // optional [N]: set to step
};

struct PolicyArgs {
  Batch b;
  int32_t policy;
  const uint8_t* obs;
  int64_t n;
  float* out;              // [n][NA+1]
  int32_t M;
};

// Per-env launchers (defined in rollout_<env>.cu).
#define AHT_DECLARE_ENV_LAUNCHERS(name)                                          \
  cudaError_t name##_ppo(const PpoArgs&, int grid, size_t smem, cudaStream_t);    \
  cudaError_t name##_xplay(const XpArgs&, int grid, size_t smem, cudaStream_t);   \
  cudaError_t name##_forced(const ForcedArgs&, cudaStream_t);                     \
  cudaError_t name##_reset(const ResetArgs&, cudaStream_t);                       \
  int name##_state_words();                                                      \
  int name##_state_bytes();                                                      \
  cudaError_t name##_set_smem_limit(size_t bytes);                                \
  int name##_occupancy(int which /* 0 PPO, 1 cross-play */, size_t smem);

AHT_DECLARE_ENV_LAUNCHERS(lbf)
AHT_DECLARE_ENV_LAUNCHERS(overcooked)
AHT_DECLARE_ENV_LAUNCHERS(hanabi)
AHT_DECLARE_ENV_LAUNCHERS(minihanabi)

// Tensor-core rollout (rollout_lbf.cu): LBF grids whose padded observation fits 256 bf16
// columns of tensor memory; PPO collection (grid = tile table entries) and cross-play
// (grid = pairs x tpp).  a.tc.split selects the fp32 (split-weight) variant.
cudaError_t lbf_ppo_tc(const PpoTcArgs&, int grid, size_t smem, cudaStream_t);
// plain collection with a dense first layer, one warp group per agent (rollout_lbf2.cu)
cudaError_t lbf_ppo_tc2(const PpoTcArgs&, int grid, size_t smem, cudaStream_t);
cudaError_t lbf_xplay_tc2(const PpoTcArgs&, int grid, size_t smem, cudaStream_t);
cudaError_t lbf_xplay_tc(const PpoTcArgs&, int grid, size_t smem, cudaStream_t);

// Streamed tensor-core cross-play step (rollout_overcooked.cu, rollout_hanabi.cu).
// grid = the launch's tiles (xp_tc_tiles), smem = xp_tc_smem_bytes.
cudaError_t overcooked_xplay_tc(const XpTcArgs&, int grid, size_t smem, cudaStream_t);
cudaError_t hanabi_xplay_tc(const XpTcArgs&, int grid, size_t smem, cudaStream_t);
cudaError_t overcooked_xplay_tc_smem_limit(size_t smem);  // once per device, before launches
cudaError_t hanabi_xplay_tc_smem_limit(size_t smem);
cudaError_t minihanabi_xplay_tc(const XpTcArgs&, int grid, size_t smem, cudaStream_t);
// test hook: the cross-play kernel's observation rows of a state array (see xplay_tc.cuh)
cudaError_t hanabi_obs_words(const uint32_t* state, int64_t n, const DevEnv& env, int seat, int words,
                             uint32_t* out, cudaStream_t s);
cudaError_t minihanabi_obs_words(const uint32_t* state, int64_t n, const DevEnv& env, int seat, int words,
                                 uint32_t* out, cudaStream_t s);
cudaError_t overcooked_obs_words(const uint32_t* state, int64_t n, const DevEnv& env, int seat, int words,
                                 uint32_t* out, cudaStream_t s);
cudaError_t minihanabi_xplay_tc_smem_limit(size_t smem);
size_t xp_tc_smem_bytes(const WideDims& w);
size_t xp_tc_state_bytes(const WideDims& w);  // room for the tile's env states (operand region)

// misc.cu
cudaError_t launch_group(const GroupArgs&, cudaStream_t);          // one-member pool
cudaError_t launch_teammate_draw(const GroupArgs&, cudaStream_t);  // kidx, hist, teammate
cudaError_t launch_policy(const PolicyArgs&, int grid, size_t smem, cudaStream_t);
cudaError_t policy_set_smem_limit(size_t bytes);
cudaError_t launch_tanh_probe(const float* x, float* y, int64_t n, cudaStream_t);
cudaError_t launch_expire_wait(uint32_t* status, uint64_t limit_ns, cudaStream_t);
int group_tiles(int64_t n_envs, int M);  // tile-table entries of a one-member-pool launch
cudaError_t launch_resample_group(const ResampleGroupArgs&, cudaStream_t);
int resample_tiles(int64_t n_envs, int M, int pool_size);  // tile-table entries, per-episode mode
// kidx[e] = pool index of env e's episode teammate, hist[k] += envs with index k
cudaError_t launch_resample_init(const Key& key, int64_t n_envs, const uint32_t* ep_step,
                                 int32_t pool_size, uint8_t* kidx, int32_t* hist, cudaStream_t);
cudaError_t launch_gae(const float* r, const float* v, const uint8_t* d, const float* v_last,
                       int64_t n, int32_t T, float gamma, float lambda, float* adv, float* tgt,
                       cudaStream_t);
cudaError_t launch_xp_reduce(const float* returns, int64_t n_pairs, int32_t P, float* matrix,
                             cudaStream_t);

// PPO ego update (ppo_update.cu).  Actor-critic ego obs_dim -> 128 -> 128 -> n_act + 1.
constexpr int kPpoTile = 64;        // samples per tile of the gradient kernel
constexpr int kPpoKP = 208;         // padded input width (obs_dim <= 207, the bias column)
constexpr int kPpoHidden = 128;
constexpr int kPpoMaxOut = 8;       // n_act + 1 <= 8
constexpr int kPpoStatBlocks = 64;  // blocks per minibatch of the advantage statistics
// packed block (bytes): W1 bf16 canonical [128][208], W2 bf16 canonical [128][128], W3 as
// two bf16 canonical [16][128] (hi, lo; rows past n_act + 1 zero), b1 [128], b2 [128],
// b3 [8] fp32
constexpr uint32_t kPkW1 = 0, kPkW2 = 53248, kPkW3hi = 86016, kPkW3lo = 90112, kPkB1 = 94208,
                   kPkB2 = 94720, kPkB3 = 95232, kPpoPackedBytes = 95264;
struct PpoLayout {  // flat parameter vector: W1 [128][D], b1, W2 [128][128], b2, W3 [O][128], b3
  int32_t D, O;
  int64_t n_params, ob1, oW2, ob2, oW3, ob3;
};
struct PpoGradArgs {
  const uint8_t* packed;
  const uint8_t* obs;       // [S][D]
  const uint8_t* act;       // [S]
  const float *logp, *val, *adv, *tgt;
  int32_t D, n_act;
  uint32_t S;               // samples
  int32_t w;                // permutation bits
  Key key;                  // permutation key
  uint32_t epoch;           // permutation counter
  uint32_t B, mb;           // samples per minibatch, minibatch index
  const float* mbstat;      // [2]: mean, 1 / (std + 1e-8) of the minibatch's advantages
  float clip_eps, vf_coef, ent_coef;
  float* partials;          // [grid][part_stride]: gradient partials, then 6 loss sums
  int64_t part_stride, n_params, oW1, ob1, oW2, ob2, oW3, ob3;
  uint32_t* status;
};
struct PpoAdamArgs {
  PpoLayout L;
  double* grad;     // [n_params] written by the reduction
  double* blocksq;  // [n_blocks] squared-norm partials
  int32_t n_blocks;
  float *params, *m, *v;
  uint8_t* packed;
  float lr, b1, b2, eps, c1, c2, max_grad_norm;
};
size_t ppo_grad_smem_bytes();
cudaError_t ppo_grad_set_smem();
cudaError_t launch_ppo_grad(const PpoGradArgs&, int grid, cudaStream_t);
cudaError_t launch_ppo_advstat(const float* adv, uint32_t S, int w, Key key, uint32_t epoch0, int E,
                               int M, uint32_t B, double* part, float* mbstat, cudaStream_t);
cudaError_t launch_ppo_pack(const PpoLayout&, const float* params, uint8_t* packed, cudaStream_t);
// Sums the partials (grad, blocksq, stats[6] = means), then (step) clips and takes the Adam step.
cudaError_t launch_f64_to_f32(const double* x, float* y, int64_t n, cudaStream_t);
cudaError_t launch_ppo_reduce_adam(const float* partials, int G, int64_t stride, const PpoAdamArgs&,
                                   float* stats, float inv_b, bool step, cudaStream_t);

// Cross-play matrix consumers (misc.cu): one CTA; n_ego, n_tm <= kXpStatsMax.
constexpr int kXpStatsMax = 2048;
struct XpStatsArgs {
  const float* xp;  // [n_ego][n_tm]
  int32_t n_ego, n_tm;
  float* upper;     // [n_tm] in/out
  float *norm, *regret, *j_aht, *j_norm, *max_regret, *brdiv;  // each may be null
  int32_t* worst;
};
cudaError_t launch_xp_stats(const XpStatsArgs&, cudaStream_t);

}  // namespace aht
