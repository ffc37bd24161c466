// rollout_impl.cuh -- fused persistent rollout kernels, templated on the env rules.
//
// One CTA owns a tile of M envs for the whole call.  Env state lives in shared memory
// from the first step to the last; each step the CTA builds the observations of its
// envs in shared memory, runs the acting policies' MLPs over the tile, samples actions
// with Philox draws, steps the envs and streams the trajectory out.  Nothing but the
// trajectory (PPO) or the final returns (cross-play) goes back to HBM.
#pragma once
#include "kernels.h"
#include "mlp_simt.cuh"

namespace aht {

struct SmemLayout {
  int64_t st, X, H1, H2, Z, envid, act, lp, val, alive, steps, list, total;
};

__host__ __device__ inline SmemLayout smem_layout(int M, const MlpDims& m, int state_bytes) {
  SmemLayout L;
  int64_t o = 0;
  L.st = o;    o = align_up(o + (int64_t)M * state_bytes, 16);
  L.X = o;     o = align_up(o + (int64_t)M * m.KP, 16);
  L.H1 = o;    o = align_up(o + (int64_t)M * m.H0 * 4, 16);
  L.H2 = o;    o = align_up(o + (int64_t)M * m.H1 * 4, 16);
  L.Z = o;     o = align_up(o + (int64_t)M * m.NOP * 4, 16);
  L.envid = o; o = align_up(o + (int64_t)M * 4, 16);
  L.act = o;   o = align_up(o + (int64_t)M * 2, 16);
  L.lp = o;    o = align_up(o + (int64_t)M * 4, 16);
  L.val = o;   o = align_up(o + (int64_t)M * 4, 16);
  L.alive = o; o = align_up(o + (int64_t)M * 4, 16);
  L.steps = o; o = align_up(o + (int64_t)M * 4, 16);
  L.list = o;  o = align_up(o + (m.sparse ? (int64_t)M * kSparseCap * 4 : 0), 16);
  L.total = o;
  return L;
}

// All of an env's state words are requested at once (one memory latency, not one per
// word): the loads complete into registers before any is stored.
template <class S>
__device__ __forceinline__ void load_state(const uint32_t* __restrict__ g, int64_t n, int64_t e,
                                           S& s) {
  constexpr int kW = (int)(sizeof(S) / 4);
  uint32_t v[kW];
#pragma unroll
  for (int w = 0; w < kW; ++w) v[w] = __ldg(g + (int64_t)w * n + e);
  uint32_t* p = reinterpret_cast<uint32_t*>(&s);
#pragma unroll
  for (int w = 0; w < kW; ++w) p[w] = v[w];
}

template <class S>
__device__ __forceinline__ void store_state(uint32_t* __restrict__ g, int64_t n, int64_t e,
                                            const S& s) {
  const uint32_t* p = reinterpret_cast<const uint32_t*>(&s);
#pragma unroll
  for (int w = 0; w < (int)(sizeof(S) / 4); ++w) g[(int64_t)w * n + e] = p[w];
}

// Copies `count` observation rows (row i of X goes to dst row ids[i]) as 32-bit words.
__device__ __forceinline__ void copy_obs_rows(const uint8_t* X, int KP, int count,
                                              const int32_t* ids, uint8_t* dst, int obs_dim) {
  const int wpr = obs_dim >> 2;
  uint32_t* d = reinterpret_cast<uint32_t*>(dst);
  for (int idx = threadIdx.x; idx < count * wpr; idx += blockDim.x) {
    const int i = idx / wpr, w = idx - i * wpr;
    d[(int64_t)ids[i] * wpr + w] = reinterpret_cast<const uint32_t*>(X + i * KP)[w];
  }
}

// ---- PPO rollout collection ------------------------------------------------------------
template <class Env>
__global__ void __launch_bounds__(kThreads) ppo_kernel(const PpoArgs a) {
  using State = typename Env::State;
  extern __shared__ __align__(16) uint8_t smem[];
  const int4 tile = a.tiles[blockIdx.x];
  const int count = tile.y;
  if (count == 0) return;
  const int M = a.M;
  const MlpDims& m = a.b.mlp;
  const SmemLayout L = smem_layout(M, m, sizeof(State));
  State* st = reinterpret_cast<State*>(smem + L.st);
  uint8_t* X = smem + L.X;
  float* H1 = reinterpret_cast<float*>(smem + L.H1);
  float* H2 = reinterpret_cast<float*>(smem + L.H2);
  float* Z = reinterpret_cast<float*>(smem + L.Z);
  int32_t* envid = reinterpret_cast<int32_t*>(smem + L.envid);
  uint8_t* act = smem + L.act;
  float* lp = reinterpret_cast<float*>(smem + L.lp);
  float* val = reinterpret_cast<float*>(smem + L.val);
  const int tid = threadIdx.x;
  const int64_t N = a.n_envs;
  const int od = a.b.env.obs_dim;

  for (int i = tid; i < M; i += blockDim.x) {
    if (i < count) {
      const int env = a.perm[tile.x + i];
      envid[i] = env;
      load_state(a.state, N, env, st[i]);
    }
    uint32_t* row = reinterpret_cast<uint32_t*>(X + i * m.KP);
    for (int w = 0; w < (m.KP >> 2); ++w) row[w] = 0u;  // padding columns stay zero
  }
  __syncthreads();
  const float* w_pol[2] = {a.b.weights + (int64_t)a.ego * m.stride,
                           a.b.weights + (int64_t)tile.z * m.stride};

  for (int t = 0; t < a.T; ++t) {
    const uint32_t gt = a.step0 + (uint32_t)t;
    for (int seat = 0; seat < 2; ++seat) {
      for (int i = tid; i < count; i += blockDim.x) Env::obs(a.b.env, st[i], seat, X + i * m.KP);
      __syncthreads();
      if (seat == 0 && a.traj.obs)
        copy_obs_rows(X, m.KP, count, envid, a.traj.obs + (int64_t)t * N * od, od);
      if (seat == 1 && a.traj1.obs)
        copy_obs_rows(X, m.KP, count, envid, a.traj1.obs + (int64_t)t * N * od, od);
      mlp_tile(w_pol[seat], m, X, H1, H2, Z, M, reinterpret_cast<uint32_t*>(smem + L.list), count);
      for (int i = tid; i < count; i += blockDim.x) {
        const float u = u01(draw0(a.b.key, (uint32_t)envid[i], gt, kStreamAct0 + seat));
        float logp;
        const int ai = sample_row(Z + i * m.NOP, m.NA, 0xFFFFFFFFu >> (32 - m.NA), u, logp);
        act[i * 2 + seat] = (uint8_t)ai;
        if (seat == 0) {
          lp[i] = logp;
          val[i] = Z[i * m.NOP + m.NA];
        } else {
          const int64_t o = (int64_t)t * N + envid[i];
          if (a.traj1.logp) a.traj1.logp[o] = logp;
          if (a.traj1.values) a.traj1.values[o] = Z[i * m.NOP + m.NA];
        }
      }
      __syncthreads();
    }
    for (int i = tid; i < count; i += blockDim.x) {
      const int env = envid[i];
      float r0, r1, team;
      const int done = Env::step(a.b.env, st[i], act[2 * i], act[2 * i + 1], r0, r1, team);
      const int64_t o = (int64_t)t * N + env;
      if (a.traj.actions) a.traj.actions[o] = act[2 * i];
      if (a.traj.tm_actions) a.traj.tm_actions[o] = act[2 * i + 1];
      if (a.traj.logp) a.traj.logp[o] = lp[i];
      if (a.traj.values) a.traj.values[o] = val[i];
      if (a.traj.rewards) a.traj.rewards[o] = team;
      if (a.traj.dones) a.traj.dones[o] = (uint8_t)(done > 0);
      if (a.traj1.actions) a.traj1.actions[o] = act[2 * i + 1];
      if (a.traj1.tm_actions) a.traj1.tm_actions[o] = act[2 * i];
      if (a.traj1.rewards) a.traj1.rewards[o] = team;
      if (a.traj1.dones) a.traj1.dones[o] = (uint8_t)(done > 0);
      if (done > 0) {
        Env::reset(a.b.env, a.b.key, (uint32_t)env, gt + 1, st[i]);
        if (a.ep_step) a.ep_step[env] = gt + 1;
      }
    }
    __syncthreads();
  }
  // Bootstrap value V_T of the state after the last step.
  if (a.traj.last_value) {
    for (int i = tid; i < count; i += blockDim.x) Env::obs(a.b.env, st[i], 0, X + i * m.KP);
    __syncthreads();
    mlp_tile(w_pol[0], m, X, H1, H2, Z, M, reinterpret_cast<uint32_t*>(smem + L.list), count);
    for (int i = tid; i < count; i += blockDim.x) a.traj.last_value[envid[i]] = Z[i * m.NOP + m.NA];
    __syncthreads();
  }
  if (a.traj1.last_value) {  // seat 1's V_T (IPPO)
    for (int i = tid; i < count; i += blockDim.x) Env::obs(a.b.env, st[i], 1, X + i * m.KP);
    __syncthreads();
    mlp_tile(w_pol[1], m, X, H1, H2, Z, M, reinterpret_cast<uint32_t*>(smem + L.list), count);
    for (int i = tid; i < count; i += blockDim.x) a.traj1.last_value[envid[i]] = Z[i * m.NOP + m.NA];
  }
  for (int i = tid; i < count; i += blockDim.x) store_state(a.state, N, envid[i], st[i]);
}

// ---- cross-play evaluation --------------------------------------------------------------
template <class Env>
__global__ void __launch_bounds__(kThreads) xplay_kernel(const XpArgs a) {
  using State = typename Env::State;
  extern __shared__ __align__(16) uint8_t smem[];
  const int M = a.M;
  const MlpDims& m = a.b.mlp;
  const SmemLayout L = smem_layout(M, m, sizeof(State));
  State* st = reinterpret_cast<State*>(smem + L.st);
  uint8_t* X = smem + L.X;
  float* H1 = reinterpret_cast<float*>(smem + L.H1);
  float* H2 = reinterpret_cast<float*>(smem + L.H2);
  float* Z = reinterpret_cast<float*>(smem + L.Z);
  uint8_t* act = smem + L.act;
  int32_t* alive = reinterpret_cast<int32_t*>(smem + L.alive);
  int32_t* nsteps = reinterpret_cast<int32_t*>(smem + L.steps);
  const int tid = threadIdx.x;

  const int pair = blockIdx.x / a.tiles_per_pair;
  const int first = (blockIdx.x - pair * a.tiles_per_pair) * M;
  const int count = min(M, a.P - first);
  const int64_t e0 = (int64_t)pair * a.P + first;
  const int64_t n_total = (int64_t)a.n_ego * a.n_tm * a.P;
  const float* w_pol[2] = {a.b.weights + (int64_t)a.ego_ids[pair / a.n_tm] * m.stride,
                           a.b.weights + (int64_t)a.tm_ids[pair % a.n_tm] * m.stride};

  for (int i = tid; i < M; i += blockDim.x) {
    if (i < count) Env::reset(a.b.env, a.b.key, (uint32_t)(e0 + i), a.step0, st[i]);
    alive[i] = i < count;
    nsteps[i] = 0;
    uint32_t* row = reinterpret_cast<uint32_t*>(X + i * m.KP);
    for (int w = 0; w < (m.KP >> 2); ++w) row[w] = 0u;
  }
  __syncthreads();

  for (int s = 0; s < a.max_steps; ++s) {
    if (!__syncthreads_or(tid < count && alive[tid])) break;
    const uint32_t gt = a.step0 + (uint32_t)s;
    const int actor = Env::kTurnBased ? (s & 1) : -1;
    for (int seat = 0; seat < 2; ++seat) {
      if (actor >= 0 && seat != actor) continue;
      for (int i = tid; i < count; i += blockDim.x)
        if (alive[i]) Env::obs(a.b.env, st[i], seat, X + i * m.KP);
      __syncthreads();
      mlp_tile(w_pol[seat], m, X, H1, H2, Z, M, reinterpret_cast<uint32_t*>(smem + L.list), count);
      for (int i = tid; i < count; i += blockDim.x) {
        if (!alive[i]) continue;
        uint32_t legal = 0xFFFFFFFFu >> (32 - m.NA);
        if (Env::kTurnBased) {
          legal = Env::legal(st[i]);
          if (Env::actor(st[i]) != seat) atomicOr(a.b.status, kStatusActorMismatch);
        }
        const float u = u01(draw0(a.b.key, (uint32_t)(e0 + i), gt, kStreamAct0 + seat));
        float logp;
        act[i * 2 + seat] = (uint8_t)sample_row(Z + i * m.NOP, m.NA, legal, u, logp);
      }
      __syncthreads();
    }
    for (int i = tid; i < count; i += blockDim.x) {
      const int64_t e = e0 + i;
      // (the host pre-fills the optional action record with 255 = no action)
      uint8_t* rec = a.actions ? a.actions + ((int64_t)s * n_total + e) * 2 : nullptr;
      if (!alive[i]) continue;
      const int a0 = (actor < 0 || actor == 0) ? act[2 * i] : 0;
      const int a1 = (actor < 0 || actor == 1) ? act[2 * i + 1] : 0;
      if (rec) {
        rec[0] = (actor < 0 || actor == 0) ? (uint8_t)a0 : 255;
        rec[1] = (actor < 0 || actor == 1) ? (uint8_t)a1 : 255;
      }
      float r0, r1, team;
      const int done = Env::step(a.b.env, st[i], a0, a1, r0, r1, team);
      if (done < 0) {
        atomicOr(a.b.status, kStatusIllegalAction);
        alive[i] = 0;
        continue;
      }
      nsteps[i] += 1;
      if (done) alive[i] = 0;
    }
    __syncthreads();
  }
  for (int i = tid; i < count; i += blockDim.x) {
    a.returns[e0 + i] = Env::ret(st[i]);
    if (a.steps) a.steps[e0 + i] = nsteps[i];
  }
}

// ---- forced step, reset, policy forward --------------------------------------------------
template <class Env>
__global__ void forced_kernel(const ForcedArgs a) {
  using State = typename Env::State;
  const int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (e >= a.n_envs) return;
  State s;
  load_state(a.state, a.n_envs, e, s);
  float r0, r1, team;
  int done = Env::step(a.b.env, s, a.actions[2 * e], a.actions[2 * e + 1], r0, r1, team);
  if (done < 0) {
    atomicOr(a.b.status, kStatusIllegalAction);
    load_state(a.state, a.n_envs, e, s);
    done = 0;
    r0 = r1 = team = 0.0f;
  }
  if (done) {
    Env::reset(a.b.env, a.b.key, (uint32_t)e, a.step + 1, s);
    if (a.ep_step) a.ep_step[e] = a.step + 1;
  }
  if (a.rewards) { a.rewards[2 * e] = r0; a.rewards[2 * e + 1] = r1; }
  if (a.team) a.team[e] = team;
  if (a.dones) a.dones[e] = (uint8_t)done;
  if (a.obs) {
    const int od = a.b.env.obs_dim;
    Env::obs(a.b.env, s, 0, a.obs + (2 * e) * od);
    Env::obs(a.b.env, s, 1, a.obs + (2 * e + 1) * od);
  }
  store_state(a.state, a.n_envs, e, s);
}

template <class Env>
__global__ void reset_kernel(const ResetArgs a) {
  using State = typename Env::State;
  const int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (e >= a.n_envs) return;
  State s;
  Env::reset(a.b.env, a.b.key, (uint32_t)e, a.step, s);
  store_state(a.state, a.n_envs, e, s);
  if (a.ep_step) a.ep_step[e] = a.step;
}

template <class Env>
struct Launch {
  using State = typename Env::State;
  static cudaError_t ppo(const PpoArgs& a, int grid, size_t smem, cudaStream_t s) {
    ppo_kernel<Env><<<grid, kThreads, smem, s>>>(a);
    return cudaGetLastError();
  }
  static cudaError_t xplay(const XpArgs& a, int grid, size_t smem, cudaStream_t s) {
    xplay_kernel<Env><<<grid, kThreads, smem, s>>>(a);
    return cudaGetLastError();
  }
  static cudaError_t forced(const ForcedArgs& a, cudaStream_t s) {
    const int blocks = (int)((a.n_envs + 127) / 128);
    forced_kernel<Env><<<blocks, 128, 0, s>>>(a);
    return cudaGetLastError();
  }
  static cudaError_t reset(const ResetArgs& a, cudaStream_t s) {
    const int blocks = (int)((a.n_envs + 127) / 128);
    reset_kernel<Env><<<blocks, 128, 0, s>>>(a);
    return cudaGetLastError();
  }
  static cudaError_t smem_limit(size_t bytes) {
    cudaError_t e = cudaFuncSetAttribute(ppo_kernel<Env>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
    if (e != cudaSuccess) return e;
    return cudaFuncSetAttribute(xplay_kernel<Env>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
  }
};

#define AHT_DEFINE_ENV_LAUNCHERS(name, EnvT)                                                   \
  cudaError_t name##_ppo(const PpoArgs& a, int g, size_t sm, cudaStream_t s) {                  \
    return Launch<EnvT>::ppo(a, g, sm, s);                                                     \
  }                                                                                            \
  cudaError_t name##_xplay(const XpArgs& a, int g, size_t sm, cudaStream_t s) {                 \
    return Launch<EnvT>::xplay(a, g, sm, s);                                                   \
  }                                                                                            \
  cudaError_t name##_forced(const ForcedArgs& a, cudaStream_t s) { return Launch<EnvT>::forced(a, s); } \
  cudaError_t name##_reset(const ResetArgs& a, cudaStream_t s) { return Launch<EnvT>::reset(a, s); }    \
  int name##_state_words() { return (int)(sizeof(EnvT::State) / 4); }                          \
  int name##_state_bytes() { return (int)sizeof(EnvT::State); }                                \
  cudaError_t name##_set_smem_limit(size_t b) { return Launch<EnvT>::smem_limit(b); }            \
  int name##_occupancy(int which, size_t sm) {                                                 \
    int n = 0;                                                                                 \
    if (which == 0) cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, ppo_kernel<EnvT>, kThreads, sm); \
    else cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, xplay_kernel<EnvT>, kThreads, sm);  \
    cudaGetLastError();                                                                        \
    return n;                                                                                  \
  }

}  // namespace aht
