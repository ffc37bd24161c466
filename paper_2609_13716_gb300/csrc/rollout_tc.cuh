// rollout_tc.cuh -- fused PPO rollout with the policy MLPs on tcgen05 tensor cores.
//
// One CTA (256 threads) owns a tile of up to 128 envs that share one teammate policy,
// for all T steps.  Per step and agent (ego = seat 0, teammate = seat 1):
//   obs (u8, shared memory) -> A operand in tensor memory (bf16, exact for small ints)
//   L1: D = X W1^T                      (M = 128 envs, N = hidden0, K = obs_dim padded)
//   epilogue: h = tanh(D + b1) split as h = hi + lo (two bf16) back into tensor memory
//   L2: D = hi W2^T + lo W2^T           (the split keeps ~2^-17 relative precision)
//   epilogue as above -> L3: z = hi W3^T + lo W3^T (logits, + value row for the ego)
//   sampling, env step and the trajectory write happen in the thread that owns the env.
// Weights (bf16, canonical K-major layout) are copied once per CTA into shared memory
// with bulk (TMA) copies; biases stay fp32.  Thread 0 issues all MMAs; the ego and
// teammate chains are interleaved so one agent's tensor-core work overlaps the other
// agent's CUDA-core epilogue.  Every mbarrier wait is bounded: on expiry the CTA
// records kStatusTimeout, drains its own MMAs (bounded), frees tensor memory and exits.
//
// Tensor memory (512 columns): agent a uses columns [256a, 256a + 128) for its A operand
// (X, then hi|lo of h1, then hi|lo of h2) and [256a + 128, 256a + 256) for its fp32
// accumulator.
#pragma once
#include "kernels.h"
#include "rollout_impl.cuh"
#include "tc_common.cuh"

namespace aht {

template <class Env>
__global__ void __launch_bounds__(256, 1) ppo_tc_kernel(const PpoTcArgs a) {
  using State = typename Env::State;
  extern __shared__ __align__(16) uint8_t smem[];  // no-swizzle operands need 16 B
  __shared__ __align__(8) uint64_t mbar[8];  // [3*agent + layer], [6] weights, [7] drain
  __shared__ uint32_t tmem_slot;

  const int4 tile = a.tiles[blockIdx.x];
  const int count = tile.y;
  if (count == 0) return;
  const TcDims& d = a.tc;
  const int tid = threadIdx.x, warp = tid >> 5, half = warp >> 2, row = tid & 127;
  const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;
  const int64_t N = a.n_envs;
  const int od = a.b.env.obs_dim;
  const int NA = a.b.mlp.NA;

  uint8_t* sW[2] = {smem, smem + d.pol_bytes};
  uint8_t* sObs = smem + 2 * d.pol_bytes;                                   // [128][KP] u8
  State* st = reinterpret_cast<State*>(sObs + 128 * d.KP);                  // [128]
  int32_t* envid = reinterpret_cast<int32_t*>(reinterpret_cast<uint8_t*>(st) + align_up(128 * sizeof(State), 16));

  if (tid == 0) {
    for (int i = 0; i < 8; ++i) tc::mbar_init(&mbar[i], 1);
    tc::mbar_init_fence();
  }
  if (warp == 0) tc::tmem_alloc(&tmem_slot, 512);
  for (int i = tid; i < 32 * d.KP; i += blockDim.x) reinterpret_cast<uint32_t*>(sObs)[i] = 0u;
  if (tid < count) {
    const int env = a.perm[tile.x + tid];
    envid[tid] = env;
    load_state(a.state, N, env, st[tid]);
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = tmem_slot;
  const int pol[2] = {a.ego, tile.z};
  if (tid == 0) {
    tc::mbar_expect_tx(&mbar[6], 2u * d.pol_bytes);
    for (int p = 0; p < 2; ++p) {
      const uint8_t* src = a.tcw + (int64_t)pol[p] * d.pol_bytes;
      for (uint32_t off = 0; off < d.pol_bytes; off += 32768u)
        tc::bulk_g2s(sW[p] + off, src + off, min(32768u, d.pol_bytes - off), &mbar[6]);
    }
  }
  bool bad = !tc::mbar_wait(&mbar[6], 0);
  uint32_t phase[6] = {0, 0, 0, 0, 0, 0};
  const uint32_t idesc_h0 = tc::idesc_bf16(128, d.H0), idesc_h1 = tc::idesc_bf16(128, d.H1);
  const uint32_t idesc_o = tc::idesc_bf16(128, d.N3);

  auto colP = [&](int ag) { return tmem + (uint32_t)(ag * 256); };
  auto colQ = [&](int ag) { return tmem + (uint32_t)(ag * 256 + 128); };
  auto bias = [&](int ag, uint32_t off) { return reinterpret_cast<const float*>(sW[ag] + off); };

  // ---- MMA issue (thread 0) ----------------------------------------------------------
  auto issue_layer = [&](int ag, int layer) {
    tc::fence_after_sync();
    const uint32_t wbase = tc::smem_u32(sW[ag]);
    if (layer == 0) {
      const uint32_t sbo = (uint32_t)(d.KP / 8) * 128u;
      for (int ks = 0; ks < d.KP / 16; ++ks)
        tc::mma_ts(colQ(ag), colP(ag) + ks * 8, tc::smem_desc(wbase + d.oW1 + ks * 256u, 128u, sbo),
                   idesc_h0, ks > 0);
    } else {
      const int K = layer == 1 ? d.H0 : d.H1;
      const uint32_t woff = layer == 1 ? d.oW2 : d.oW3;
      const uint32_t idesc = layer == 1 ? idesc_h1 : idesc_o;
      const uint32_t sbo = (uint32_t)(K / 8) * 128u;
      for (int part = 0; part < 2; ++part)  // hi, then lo half of the split activations
        for (int ks = 0; ks < K / 16; ++ks)
          tc::mma_ts(colQ(ag), colP(ag) + part * (K / 2) + ks * 8,
                     tc::smem_desc(wbase + woff + ks * 256u, 128u, sbo), idesc, (part | ks) != 0);
    }
    tc::commit(&mbar[3 * ag + layer]);
  };

  // ---- observation tile -> tensor memory (both halves, 8 columns per chunk) -----------
  auto write_x = [&](int ag) {
    const int chunks = d.KP / 16, first = half ? (chunks + 1) / 2 : 0, last = half ? chunks : (chunks + 1) / 2;
    const uint8_t* rowp = sObs + row * d.KP;
    for (int c = first; c < last; ++c) {
      const uint4 q = *reinterpret_cast<const uint4*>(rowp + 16 * c);
      const uint32_t w4[4] = {q.x, q.y, q.z, q.w};
      uint32_t v[8];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const uint32_t x = w4[j];
        v[2 * j] = tc::pack_bf16((float)(x & 0xFFu), (float)((x >> 8) & 0xFFu));
        v[2 * j + 1] = tc::pack_bf16((float)((x >> 16) & 0xFFu), (float)(x >> 24));
      }
      tc::st_x8(colP(ag) + lane_base + 8 * c, v);
    }
    tc::wait_st();
  };

  // ---- hidden-layer epilogue: tanh(D + b), split into bf16 hi | lo -> A operand -------
  auto epilogue = [&](int ag, int layer) {
    const int H = layer == 0 ? d.H0 : d.H1;
    const float* b = bias(ag, layer == 0 ? d.ob1 : d.ob2);
    for (int c0 = half * (H / 2); c0 < (half + 1) * (H / 2); c0 += 32) {
      uint32_t v[32];
      tc::ld_x32(colQ(ag) + lane_base + c0, v);
      tc::wait_ld();
      uint32_t hi[16], lo[16];
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        const float h0 = tanhf(__uint_as_float(v[2 * j]) + b[c0 + 2 * j]);
        const float h1 = tanhf(__uint_as_float(v[2 * j + 1]) + b[c0 + 2 * j + 1]);
        const __nv_bfloat16 a0 = __float2bfloat16_rn(h0), a1 = __float2bfloat16_rn(h1);
        hi[j] = (uint32_t)__bfloat16_as_ushort(a0) | ((uint32_t)__bfloat16_as_ushort(a1) << 16);
        lo[j] = tc::pack_bf16(h0 - __bfloat162float(a0), h1 - __bfloat162float(a1));
      }
      tc::st_x16(colP(ag) + lane_base + c0 / 2, hi);
      tc::st_x16(colP(ag) + lane_base + H / 2 + c0 / 2, lo);
    }
    tc::wait_st();
  };

  // ---- logits (warps 0-3 only): z = D + b3 ---------------------------------------------
  auto logits = [&](int ag, float (&z)[16]) {
    uint32_t v[16];
    tc::ld_x16(colQ(ag) + lane_base, v);
    tc::wait_ld();
    const float* b = bias(ag, d.ob3);
#pragma unroll
    for (int j = 0; j < 16; ++j) z[j] = __uint_as_float(v[j]) + b[j];
  };

  auto wait_layer = [&](int ag, int layer) {
    const int i = 3 * ag + layer;
    if (!tc::mbar_wait(&mbar[i], phase[i] & 1u)) bad = true;
    phase[i] += 1;
    tc::fence_after_sync();
  };
  // Barrier after which thread 0 may issue: tensor-memory traffic of all threads is done.
  auto handoff = [&]() -> bool {
    tc::fence_before_sync();
    return __syncthreads_or(bad) != 0;
  };

  if (__syncthreads_or(bad)) goto drain;

  for (int t = 0; t <= a.T; ++t) {
    const bool boot = t == a.T;  // after the last step: the ego's V_T only
    if (boot && !a.traj.last_value) break;
    const uint32_t gt = a.step0 + (uint32_t)t;
    // observations of both seats, L1 of each as soon as its tile is in tensor memory
    for (int ag = 0; ag < (boot ? 1 : 2); ++ag) {
      if (half == 0 && row < count) Env::obs(a.b.env, st[row], ag, sObs + row * d.KP);
      __syncthreads();
      if (ag == 0 && !boot && a.traj.obs)
        copy_obs_rows(sObs, d.KP, count, envid, a.traj.obs + (int64_t)t * N * od, od);
      write_x(ag);
      if (handoff()) goto drain;
      if (tid == 0) issue_layer(ag, 0);
    }
    for (int layer = 0; layer < 2; ++layer) {
      for (int ag = 0; ag < (boot ? 1 : 2); ++ag) {
        wait_layer(ag, layer);
        epilogue(ag, layer);
        if (handoff()) goto drain;
        if (tid == 0) issue_layer(ag, layer + 1);
      }
    }
    float z[16];
    int act0 = 0, act1 = 0;
    float lp0 = 0.f, val0 = 0.f;
    wait_layer(0, 2);
    if (half == 0) {
      logits(0, z);
      val0 = z[NA];
      if (boot) {
        if (row < count) a.traj.last_value[envid[row]] = val0;
      } else if (row < count) {
        const float u = u01(draw0(a.b.key, (uint32_t)envid[row], gt, kStreamAct0));
        act0 = sample_row(z, NA, 0xFFFFFFFFu >> (32 - NA), u, lp0);
      }
    }
    if (boot) break;
    wait_layer(1, 2);
    if (half == 0) {
      logits(1, z);
      if (row < count) {
        float lp1;
        const float u = u01(draw0(a.b.key, (uint32_t)envid[row], gt, kStreamAct1));
        act1 = sample_row(z, NA, 0xFFFFFFFFu >> (32 - NA), u, lp1);
        const int env = envid[row];
        float r0, r1, team;
        const int done = Env::step(a.b.env, st[row], act0, act1, r0, r1, team);
        const int64_t o = (int64_t)t * N + env;
        if (a.traj.actions) a.traj.actions[o] = (uint8_t)act0;
        if (a.traj.tm_actions) a.traj.tm_actions[o] = (uint8_t)act1;
        if (a.traj.logp) a.traj.logp[o] = lp0;
        if (a.traj.values) a.traj.values[o] = val0;
        if (a.traj.rewards) a.traj.rewards[o] = team;
        if (a.traj.dones) a.traj.dones[o] = (uint8_t)(done > 0);
        if (done > 0) Env::reset(a.b.env, a.b.key, (uint32_t)env, gt + 1, st[row]);
      }
    }
    if (handoff()) goto drain;
  }
  if (tid < count) store_state(a.state, N, envid[tid], st[tid]);

drain:
  if (__syncthreads_or(bad)) {
    if (tid == 0) atomicOr(a.b.status, kStatusTimeout);
  }
  // Wait (bounded) until every MMA this CTA issued has completed, then free tensor memory.
  if (tid == 0) {
    tc::commit(&mbar[7]);
    tc::mbar_wait(&mbar[7], 0);
  }
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 0) {
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, 512);
  }
}

template <class Env>
struct LaunchTc {
  static cudaError_t ppo(const PpoTcArgs& a, int grid, size_t smem, cudaStream_t s) {
    cudaError_t e = cudaFuncSetAttribute(ppo_tc_kernel<Env>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    ppo_tc_kernel<Env><<<grid, 256, smem, s>>>(a);
    return cudaGetLastError();
  }
};

}  // namespace aht
