// rollout_tc2.cuh -- LBF rollouts with a dense first layer (PPO collection, IPPO and
// cross-play), with the ego and the teammate on separate warp groups.
//
// One CTA owns a tile of up to 128 envs that share a teammate policy, for all T steps.
// Per step and agent (ego = seat 0, teammate = seat 1):
//   obs (u8, shared memory, a constant 1 after the last feature) -> A operand in tensor
//       memory as bf16 (exact: small integers)
//   L1 (tensor cores): D = [o 1] [W1 b1]^T      (M = 128 envs, N = hidden0, K = KP)
//   epilogue 1: r1 = 1 / (1 + exp(2 D)) split r1 = hi + lo (two bf16) into tensor memory;
//       tanh(D) = 1 - 2 r1, and the block's W2, b2 hold -2 W2 and b2 + W2 1, so L2 sees
//       exactly the tanh layer (the same for r2 and W3, b3 below)
//   L2 (tensor cores): D = hi W2'^T + lo W2'^T  (the split keeps ~2^-17 relative precision
//       of r1 with bf16 operands and fp32 accumulate)
//   epilogue 2: r2 = 1 / (1 + exp(2 (D + b2))), split again, and z = W3' r2 + b3' by
//       mma.sync m16n8k16 from registers (16x256b accumulator loads are its fragment
//       layout; a handful of outputs would waste an N = 16 tcgen05 instruction's round trip)
//   sampling, env step, trajectory write.
// Each agent has its own eight warps:
//   warps 0-7   ego group: thread r and r + 128 own env row r (tensor-memory lane r) and
//               split the ego's columns; they also step the envs and write the trajectory;
//   warps 8-15  teammate group: the same for the teammate (or its rule).
// The two agents' dependent chains (observation -> L1 -> epilogue 1 -> L2 -> epilogue 2 ->
// sampling) run concurrently, four warps per SM sub-partition.  There is no MMA warp
// (sixteen warps keep 128 registers a thread): once a group's operand is in tensor memory
// (a group barrier), its first thread issues the layer's MMAs and commits them to the
// group's accumulator barrier.  The groups share one observation buffer: the teammate's
// rows are built first, and once they are in tensor memory the buffer passes to the ego
// (an mbarrier).  Both groups meet twice per step on a named barrier that also ORs their
// error flags: once both actions exist (then the ego group's first half steps the envs
// while, for gathered tiles, the teammate group and the ego's second half write the ego's
// rows to the trajectory) and once the new state is in shared memory.  Every mbarrier wait
// is bounded (2 s): on expiry the CTA records kStatusTimeout, stops, waits (bounded) for
// its own MMAs, frees tensor memory and exits.
//
// Tensor memory (512 columns): agent a uses columns [256a, 256a + 128) for its A operand
// (X, then hi|lo of h1) and [256a + 128, 256a + 256) for its fp32 accumulator.
#pragma once
#include "rollout_tc.cuh"

namespace aht {

constexpr int kT2Group = 256;     // threads per agent group
constexpr int kT2Threads = 512;   // both groups
constexpr int kT2AllBar = 1;      // named barrier ids: both groups (OR of the error flags)
constexpr int kT2GroupBar = 2;    // 2 + g: group g
constexpr int kT2PairBar = 4;     // 4 + 4 g + q: warps 8 g + q and 8 g + q + 4 (rows 32 q ..)

// kXp: cross-play instead of collection -- a tile is up to 128 envs of one pair (ego i,
// teammate j), reset at the call's first step and frozen once its first episode ends; the
// CTA stops when every env of the tile is done and writes each env's return and length
// (NaN returns if it gave up); no trajectory.
// kIppo (collection, contiguous tiles): seat 1 learns too, and its trajectory goes to
// a.traj1 -- its log-probabilities and values from its sampling threads, its actions,
// rewards and dones from the env step, its observation rows (the ego's with the seats'
// channels swapped, Env::other_seat_word) by the row-copy warps, and its V_T.
template <class Env, bool kSplit, bool kGather, bool kXp, bool kIppo = false>
__global__ void __launch_bounds__(kT2Threads, 1) ppo2_tc_kernel(const PpoTcArgs a) {
  using State = typename Env::State;
  constexpr int NA = Env::kNumActions;
  static_assert(kT2Threads / 32 <= 24, "gather scratch: one total per warp");
  extern __shared__ __align__(16) uint8_t smem[];
  __shared__ __align__(8) uint64_t acc_bar[4];     // [2*agent + layer], tcgen05.commit
  __shared__ __align__(8) uint64_t wload_bar[2], drain_bar[2];  // per agent
  __shared__ __align__(8) uint64_t buf_free;       // teammate rows in tensor memory (256)
  __shared__ __align__(8) uint64_t never_bar;      // test hook: nothing arrives on it
  __shared__ uint32_t tmem_slot;
  const TcDims& d = a.tc;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, row = tid & 127;

  // A per-episode call launches its steps after the first as programmatic dependents of
  // the step before: everything up to griddepcontrol.wait touches nothing that step
  // writes -- the barriers, tensor memory and the ego's weights (the ego is the same for
  // the whole call).  (Without that launch attribute the wait returns at once.)
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  if (tid == 0) {
    for (int i = 0; i < 4; ++i) tc::mbar_init(&acc_bar[i], 1);
    for (int i = 0; i < 2; ++i) {
      tc::mbar_init(&wload_bar[i], 1);
      tc::mbar_init(&drain_bar[i], 1);
    }
    tc::mbar_init(&buf_free, kT2Group);
    tc::mbar_init(&never_bar, 1);
    tc::mbar_init_fence();
    // the ego's policy block -> shared memory, waited for by the ego group (collection:
    // the same ego for every tile; cross-play: once the tile is known, below)
    if (!kXp) {
      const uint8_t* src = a.tcw + (int64_t)a.ego * d.pol_bytes;
      tc::mbar_expect_tx(&wload_bar[0], d.pol_bytes);
      for (uint32_t off = 0; off < d.pol_bytes; off += 32768u)
        tc::bulk_g2s(smem + off, src + off, min(32768u, d.pol_bytes - off), &wload_bar[0]);
    }
  }
  if (warp == 0) tc::tmem_alloc(&tmem_slot, 512);
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  asm volatile("griddepcontrol.wait;" ::: "memory");

  int32_t* const rowenv = kGather ? reinterpret_cast<int32_t*>(smem + a.g.scratch_off) : nullptr;
  static_assert(!(kXp && kGather), "cross-play tiles are contiguous");
  static_assert(!(kIppo && (kXp || kGather)), "IPPO is collection on contiguous tiles");
  const TcTile tile = tc_find_tile<kXp, kGather>(a, rowenv);
  const int64_t env0 = tile.env0;
  const int count = tile.count, tm_pol = tile.tm_pol, g_k = tile.g_k;
  if (kXp && tid == 0) {  // cross-play: this tile's ego
    const uint8_t* src = a.tcw + (int64_t)tile.ego_pol * d.pol_bytes;
    tc::mbar_expect_tx(&wload_bar[0], d.pol_bytes);
    for (uint32_t off = 0; off < d.pol_bytes; off += 32768u)
      tc::bulk_g2s(smem + off, src + off, min(32768u, d.pol_bytes - off), &wload_bar[0]);
  }
  if (count <= 0) {  // no rows: the ego's copy lands, then tensor memory is freed
    if (tid == 0) tc::mbar_wait(&wload_bar[0], 0);
    tc::fence_before_sync();
    __syncthreads();
    if (warp == 0) {
      tc::fence_after_sync();
      tc::tmem_dealloc(tmem_slot, 512);
    }
    return;
  }
  const bool tm_rule = tm_pol < 0;  // LBF heuristic -1 - id: no teammate network
  const int grp = warp >> 3;                 // 0 ego, 1 teammate
  const int half = (warp >> 2) & 1;          // which half of the agent's columns
  auto env_of = [&](int r) -> int64_t { return kGather ? (int64_t)rowenv[r] : env0 + r; };
  const int64_t my_env = row < count ? env_of(row) : 0;
  const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;
  const int64_t N = a.n_envs;
  const int od = a.b.env.obs_dim;
  const int cells = od / 4;
  const int chunks = d.KP / 16;
  const int split = (chunks + 1) / 2;
  const int my_c0 = half ? split : 0, my_c1 = half ? chunks : split;
  const int my_w0 = min(4 * my_c0, cells), my_w1 = min(4 * my_c1, cells);
  const bool boot1 = kIppo && tm_pol >= 0 && a.traj1.last_value != nullptr;  // seat 1's V_T
  const bool with_boot = !kXp && (a.traj.last_value != nullptr || boot1);
  const bool obs_copy = kGather && a.traj.obs != nullptr;  // 12 warps store the rows during the step

  uint8_t* const sW0 = smem;                                                // policy blocks
  uint8_t* const sObs = smem + 2 * d.pol_bytes;                             // [128][obs_dim] u8
  State* st = reinterpret_cast<State*>(sObs + align_up(128 * od, 16));      // [128]
  uint8_t* act1s = reinterpret_cast<uint8_t*>(st) + align_up(128 * sizeof(State), 16);  // [128]
  float* zpart = reinterpret_cast<float*>(act1s + 128);                     // [2][2][128][8]

  for (int i = tid; i < 32 * od; i += blockDim.x) reinterpret_cast<uint32_t*>(sObs)[i] = 0u;
  if (tid < count) {
    if constexpr (kXp) Env::reset(a.b.env, a.b.key, (uint32_t)(env0 + tid), a.step0, st[tid]);
    else load_state(a.state, N, env_of(tid), st[tid]);
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = tmem_slot;

  {
    const int ag = grp;  // the agent this thread works for
    const bool leader = (tid & (kT2Group - 1)) == 0;  // issues the group's copies and MMAs
    const bool net = ag == 0 || !tm_rule;              // the group runs a network
    bool bad = false;
    // the teammate's policy block -> shared memory (its leader; the ego's is on its way),
    // waited for by the group
    if (leader && net && ag == 1) {
      const uint8_t* src = a.tcw + (int64_t)tm_pol * d.pol_bytes;
      uint8_t* dst = sW0 + (size_t)ag * d.pol_bytes;
      tc::mbar_expect_tx(&wload_bar[ag], d.pol_bytes);
      for (uint32_t off = 0; off < d.pol_bytes; off += 32768u)
        tc::bulk_g2s(dst + off, src + off, min(32768u, d.pol_bytes - off), &wload_bar[ag]);
    }
    if (net && !tc::mbar_wait(&wload_bar[ag], 0)) bad = true;
    bad = __any_sync(0xFFFFFFFFu, bad);
    uint32_t n_issued = 0;  // MMA batches this thread committed (leaders)
    // the group's operand of `layer` is in tensor memory: its leader issues the layer.
    // Every thread of the group calls this at each operand point, whether or not it built
    // its part (its error flag set): the barrier ORs the flags, so the group agrees.
    auto issue = [&](int layer) {
      tc::fence_before_sync();
      bad = tc::bar_or(kT2GroupBar + ag, kT2Group, bad);
      if (!leader || bad) return;
      tc::fence_after_sync();
      const uint32_t wbase = tc::smem_u32(sW0) + (uint32_t)ag * d.pol_bytes;
      const uint32_t P = tmem + (uint32_t)(ag * 256), Q = P + 128;
      if (layer == 0) {
        const uint32_t idesc = tc::idesc_bf16(128, d.H0), sbo = (uint32_t)(d.KP / 8) * 128u;
        const uint64_t w0 = tc::smem_desc(wbase + d.oW1, 128u, sbo);
        for (int ks = 0; ks < d.KP / 16; ++ks) tc::mma_ts(Q, P + 8 * ks, w0 + 16u * ks, idesc, ks > 0);
        if constexpr (kSplit) {
          const uint64_t w1 = tc::smem_desc(wbase + d.oW1lo, 128u, sbo);
          for (int ks = 0; ks < d.KP / 16; ++ks) tc::mma_ts(Q, P + 8 * ks, w1 + 16u * ks, idesc, 1u);
        }
      } else {
        const uint32_t idesc = tc::idesc_bf16(128, d.H1), sbo = (uint32_t)(d.H0 / 8) * 128u;
        const uint64_t w0 = tc::smem_desc(wbase + d.oW2, 128u, sbo);
        for (int ks = 0; ks < d.H0 / 16; ++ks) tc::mma_ts(Q, P + 8 * ks, w0 + 16u * ks, idesc, ks > 0);
        for (int ks = 0; ks < d.H0 / 16; ++ks) tc::mma_ts(Q, P + d.H0 / 2 + 8 * ks, w0 + 16u * ks, idesc, 1u);
        if constexpr (kSplit) {
          const uint64_t w1 = tc::smem_desc(wbase + d.oW2lo, 128u, sbo);
          for (int ks = 0; ks < d.H0 / 16; ++ks) tc::mma_ts(Q, P + 8 * ks, w1 + 16u * ks, idesc, 1u);
        }
      }
      tc::commit(&acc_bar[2 * ag + layer]);
      n_issued += 1;
    };
    auto wait_acc = [&](int layer, uint32_t parity) {
      if (!bad && !tc::mbar_wait(&acc_bar[2 * ag + layer], parity)) bad = true;
      bad = __any_sync(0xFFFFFFFFu, bad);  // warp-uniform: tensor-memory loads are collective
      tc::fence_after_sync();
    };
    auto wait_bar = [&](uint64_t* bar, uint32_t parity) {
      if (!bad && !tc::mbar_wait(bar, parity)) bad = true;
      bad = __any_sync(0xFFFFFFFFu, bad);
    };
    // both groups; every thread leaves with the OR of the error flags
    auto sync_all = [&]() {
      bad = tc::bar_or(kT2AllBar, kT2Threads, bad);
      return bad;
    };
    auto pair_sync = [&]() { tc::bar_sync(kT2PairBar + 4 * grp + (warp & 3), 64); };
    const uint8_t* const pol_block = sW0 + (size_t)ag * d.pol_bytes;
    const uint32_t P = tmem + (uint32_t)(ag * 256) + lane_base, Q = P + 128;

    // observation (this thread's half row, built in shared memory) -> bf16 A operand of
    // L1 in tensor memory; feature obs_dim is the constant 1 that carries b1
    auto obs_x = [&](const State& s) {
      uint32_t* roww = reinterpret_cast<uint32_t*>(sObs + row * od);
      if (row < count) Env::obs_words(a.b.env, s, ag, roww, my_w0, my_w1);
      for (int c = my_c0; c < my_c1; ++c) {
        uint32_t w4[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const int w = 4 * c + j;
          w4[j] = w < cells ? roww[w] : (w == cells ? 1u : 0u);
        }
        uint32_t v[8];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          v[2 * j] = tc::bytes_to_bf16x2(w4[j], 0);
          v[2 * j + 1] = tc::bytes_to_bf16x2(w4[j], 2);
        }
        tc::st_x8(P + 8 * c, v);
      }
      tc::wait_st();
    };
    // epilogue 1: r1 = 1 / (1 + exp(2 D)) -> hi | lo bf16 A operand of L2, 32 units per
    // tensor-memory load (16 independent pairs between waits; tanh(D) = 1 - 2 r1: the
    // block's W2, b2 absorb the affine map, as W3, b3 do for r2)
    auto epilogue1 = [&]() {
      const int H = d.H0;
#pragma unroll 1
      for (int c0 = half * (H / 2); c0 < (half + 1) * (H / 2); c0 += 32) {
        uint32_t v[32];
        tc::ld_x32(Q + c0, v);
        tc::wait_ld();
        uint32_t hi[16], lo[16];
#pragma unroll
        for (int j = 0; j < 16; ++j)
          tc::split_bf16x2_p(tc::logistic2(tc::f2_mul(tc::f2_pack(__uint_as_float(v[2 * j]), __uint_as_float(v[2 * j + 1])), tc::kTwoOverLn2x2)),
                             hi[j], lo[j]);
        tc::st_x16(P + c0 / 2, hi);
        tc::st_x16(P + H / 2 + c0 / 2, lo);
      }
      tc::wait_st();
    };
    // epilogue 2: r2 = 1 / (1 + exp(2 (D + b2))) split hi + lo, and this half's partial z = W3' r2 by
    // mma.sync m16n8k16 from the 16x256b accumulator fragments (see ppo_tc_kernel)
    auto epilogue2 = [&]() {
      const int H = d.H1;
      const float* b2 = reinterpret_cast<const float*>(pol_block + d.ob2);
      const uint32_t Qq = tmem + (uint32_t)(ag * 256 + 128) + lane_base;
      const uint32_t* W3f = reinterpret_cast<const uint32_t*>(pol_block + d.oW3);
      const uint32_t* W3l = W3f + H * 4;
      const int g = lane >> 2, c4 = lane & 3;
      float zacc[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
      // two 16-unit chunks (both row groups of each) under one wait: 16 independent pairs;
      // each row group accumulates chunk by chunk, hi then lo, as in ppo_tc_kernel
#pragma unroll 1
      for (int c0 = half * (H / 2); c0 < (half + 1) * (H / 2); c0 += 32) {
        uint32_t tt[2][2][2][4];  // [chunk][row group][column half][fragment]
#pragma unroll
        for (int cc = 0; cc < 2; ++cc)
#pragma unroll
          for (int rg = 0; rg < 2; ++rg) {
            tc::ld_16x256b(Qq + ((uint32_t)(16 * rg) << 16) + (uint32_t)(c0 + 16 * cc), tt[cc][rg][0]);
            tc::ld_16x256b(Qq + ((uint32_t)(16 * rg) << 16) + (uint32_t)(c0 + 16 * cc + 8), tt[cc][rg][1]);
          }
        uint2 bw[2], bl[2];
        uint64_t bA[2], bB[2];
#pragma unroll
        for (int cc = 0; cc < 2; ++cc) {
          const int j = (c0 >> 4) + cc, u0 = c0 + 16 * cc;
          bw[cc] = *reinterpret_cast<const uint2*>(W3f + (j * 32 + lane) * 2);
          bl[cc] = make_uint2(0u, 0u);
          if constexpr (kSplit) bl[cc] = *reinterpret_cast<const uint2*>(W3l + (j * 32 + lane) * 2);
          bA[cc] = *reinterpret_cast<const uint64_t*>(b2 + u0 + 2 * c4);
          bB[cc] = *reinterpret_cast<const uint64_t*>(b2 + u0 + 8 + 2 * c4);
        }
        tc::wait_ld();
#pragma unroll
        for (int cc = 0; cc < 2; ++cc)
#pragma unroll
          for (int rg = 0; rg < 2; ++rg) {
            const uint32_t (&t0)[4] = tt[cc][rg][0];
            const uint32_t (&t1)[4] = tt[cc][rg][1];
            uint32_t ahi[4], alo[4];
            tc::split_bf16x2_p(tc::logistic2(tc::f2_fma(tc::f2_pack(__uint_as_float(t0[0]), __uint_as_float(t0[1])), tc::kTwoOverLn2x2, bA[cc])),
                               ahi[0], alo[0]);
            tc::split_bf16x2_p(tc::logistic2(tc::f2_fma(tc::f2_pack(__uint_as_float(t0[2]), __uint_as_float(t0[3])), tc::kTwoOverLn2x2, bA[cc])),
                               ahi[1], alo[1]);
            tc::split_bf16x2_p(tc::logistic2(tc::f2_fma(tc::f2_pack(__uint_as_float(t1[0]), __uint_as_float(t1[1])), tc::kTwoOverLn2x2, bB[cc])),
                               ahi[2], alo[2]);
            tc::split_bf16x2_p(tc::logistic2(tc::f2_fma(tc::f2_pack(__uint_as_float(t1[2]), __uint_as_float(t1[3])), tc::kTwoOverLn2x2, bB[cc])),
                               ahi[3], alo[3]);
            tc::mma_m16n8k16_bf16(zacc[rg], ahi, bw[cc].x, bw[cc].y);
            tc::mma_m16n8k16_bf16(zacc[rg], alo, bw[cc].x, bw[cc].y);
            if constexpr (kSplit) tc::mma_m16n8k16_bf16(zacc[rg], ahi, bl[cc].x, bl[cc].y);
          }
      }
      float* zp = zpart + (ag * 2 + half) * 128 * 8;
#pragma unroll
      for (int rg = 0; rg < 2; ++rg) {
        const int r = 32 * (warp & 3) + 16 * rg + g;
        *reinterpret_cast<float2*>(zp + r * 8 + 2 * c4) = make_float2(zacc[rg][0], zacc[rg][1]);
        *reinterpret_cast<float2*>(zp + (r + 8) * 8 + 2 * c4) = make_float2(zacc[rg][2], zacc[rg][3]);
      }
    };
    // full logits of this group's agent: (half-0 partial + half-1 partial) + b3
    auto logits = [&](float (&z)[16]) {
      const float* p0 = zpart + ((ag * 2 + 0) * 128 + row) * 8;
      const float* p1 = zpart + ((ag * 2 + 1) * 128 + row) * 8;
      const float* b3 = reinterpret_cast<const float*>(pol_block + d.ob3);
      // two 16-byte loads per half (a row's 8 partial sums; 8-byte-strided scalar loads
      // would hit the same banks 8 ways)
      const float4 a0 = *reinterpret_cast<const float4*>(p0), a1 = *reinterpret_cast<const float4*>(p0 + 4);
      const float4 c0 = *reinterpret_cast<const float4*>(p1), c1 = *reinterpret_cast<const float4*>(p1 + 4);
      const float pa[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
      const float pc[8] = {c0.x, c0.y, c0.z, c0.w, c1.x, c1.y, c1.z, c1.w};
#pragma unroll
      for (int o = 0; o < 8; ++o) z[o] = (pa[o] + pc[o]) + b3[o];
#pragma unroll
      for (int o = 8; o < 16; ++o) z[o] = 0.0f;
    };
    // test hook: this row's outputs of step t
    auto dbg_store = [&](int t, const float (&z)[16]) {
      if (!a.dbg_logits) return;
      const int64_t rows = kXp ? a.xp.n_total : N;
      float* p = a.dbg_logits + (((int64_t)t * rows + my_env) * 2 + ag) * kDbgStride;
#pragma unroll
      for (int o = 0; o < 8; ++o) p[o] = z[o];
    };
    // contiguous tiles: the ego's rows -> trajectory [t][env0 .. env0 + count) as one
    // contiguous block, by one bulk (TMA) store when 16-byte aligned, else by the group
    const bool bulk_obs = !kGather && a.traj.obs && (count * od) % 16 == 0;
    auto copy_rows_contiguous = [&](int t) {
      uint8_t* dst = a.traj.obs + ((int64_t)t * N + env0) * od;
      const uint32_t bytes = (uint32_t)(count * od);
      if (bulk_obs && (reinterpret_cast<uintptr_t>(dst) & 15u) == 0) {
        if (tid == 0) {
          tc::bulk_s2g(dst, sObs, bytes);
          tc::bulk_commit();
        }
      } else {
        const uint32_t* src = reinterpret_cast<const uint32_t*>(sObs);
        uint32_t* d32 = reinterpret_cast<uint32_t*>(dst);
        for (uint32_t w = tid; w < bytes / 4; w += kT2Group) d32[w] = src[w];
      }
    };
    // gathered tiles: the ego's rows -> their envs' trajectory rows, while the ego group's
    // first half steps the envs: the 12 warps of the teammate group and of the ego's
    // second half take the tile's count x cells words in turn (consecutive lanes,
    // consecutive words of a row; row = word / cells by a reciprocal multiply, exact for
    // fewer than 2^16 words)
    const uint32_t cells_rcp = 0xFFFFFFFFu / (uint32_t)cells + 1u;
    auto copy_rows_gathered = [&](int t, int cw) {
      constexpr int kCopyWarps = 12;
      uint32_t* const base = reinterpret_cast<uint32_t*>(a.traj.obs + (int64_t)t * N * od);
      const uint32_t* const src = reinterpret_cast<const uint32_t*>(sObs);
      const int total = count * cells;
#pragma unroll 4
      for (int f = cw * 32 + lane; f < total; f += kCopyWarps * 32) {
        const int r = (int)__umulhi((uint32_t)f, cells_rcp);
        base[(int64_t)rowenv[r] * cells + (f - r * cells)] = src[f];
      }
    };

    // Steps 0..T-1, then (if requested) the ego's V_T of the state after the last step.
    const int n_steps = kXp ? a.xp.max_steps : a.T;
    bool alive = true;  // cross-play: the row's episode is running (ego group, first half)
    int nsteps = 0;
    for (int t = 0; t <= n_steps; ++t) {
      const bool boot = t == n_steps;
      if (boot && !with_boot) break;
      if constexpr (kXp) {  // every env of the tile is done: stop (no MMA is in flight)
        if (!tc::bar_or(kT2AllBar, kT2Threads, ag == 0 && half == 0 && row < count && alive)) break;
      }
      const uint32_t par = (uint32_t)t & 1u, gt = a.step0 + (uint32_t)t;
      const bool sampler = half == 0 && row < count && !boot;
      // this step's action draw (Philox), computed while L1 runs on the tensor cores
      float u_act = 0.0f;
      auto draw_action = [&]() {
        if (sampler) u_act = u01(draw0(a.b.key, (uint32_t)my_env, gt, kStreamAct0 + ag));
      };
      const State s = st[row];  // register copy for this step (rows past count are never used)
      float z[16];
      int act0 = 0;
      float lp0 = 0.f, val0 = 0.f;
      if (ag == 1) {
        // ---------------------------- teammate group -------------------------------
        const bool run = (!boot || boot1) && !tm_rule;
        if (run) obs_x(s);
        tc::mbar_arrive(&buf_free);  // its rows are in tensor memory: the buffer is the ego's
        if (run) {
          issue(0);
          draw_action();
          wait_acc(0, par);
          if (!bad) epilogue1();
          issue(1);
          wait_acc(1, par);
          if (!bad) epilogue2();
        }
        pair_sync();
        if (sampler) {
          if (tm_rule) {
            act1s[row] = (uint8_t)Env::heuristic(a.b.env, st[row], -1 - tm_pol);  // st[row] == s
          } else {
            logits(z);
            dbg_store(t, z);
            float lp;
            act1s[row] = (uint8_t)sample_k<NA>(z, 0xFFFFFFFFu >> (32 - NA), u_act, lp);
            if constexpr (kIppo) {  // seat 1's learner fields
              const int64_t o = (int64_t)t * N + my_env;
              if (a.traj1.logp) a.traj1.logp[o] = lp;
              if (a.traj1.values) a.traj1.values[o] = z[NA];
            }
          }
        } else if (boot1 && boot && half == 0 && row < count) {  // seat 1's V_T
          logits(z);
          a.traj1.last_value[my_env] = z[NA];
        }
      } else {
        // ------------------------------- ego group ---------------------------------
        wait_bar(&buf_free, par);
        obs_x(s);
        // contiguous tiles: the rows (ordinary stores) are read by the bulk copy engine
        if (!kGather && !boot && a.traj.obs) tc::fence_proxy_async();
        issue(0);  // (its group barrier also orders the rows before the copy)
        draw_action();
        if (!kGather && !boot && a.traj.obs) copy_rows_contiguous(t);
        if (t == a.dbg_expire_step) {  // test hook: an accumulator wait that never completes
          if (!bad && !tc::mbar_wait(&never_bar, 0, a.dbg_expire_ns)) bad = true;
          bad = __any_sync(0xFFFFFFFFu, bad);
        }
        wait_acc(0, par);
        if (!bad) epilogue1();
        issue(1);
        wait_acc(1, par);
        if (!bad) epilogue2();
        pair_sync();
        if (boot) {
          if (half == 0 && row < count && a.traj.last_value) {
            logits(z);
            a.traj.last_value[my_env] = z[NA];
          }
        } else if (sampler) {
          logits(z);
          dbg_store(t, z);
          act0 = sample_k<NA>(z, 0xFFFFFFFFu >> (32 - NA), u_act, lp0);
          val0 = z[NA];
        }
      }
      if (sync_all() || boot) break;  // both actions exist
      bool stayed = false;            // per-episode gather: the env keeps its teammate
      if (kXp && ag == 0 && half == 0 && row < count && alive) {
        State s2 = s;
        const int act1 = act1s[row];
        if (a.xp.actions) {
          uint8_t* rec = a.xp.actions + ((int64_t)t * a.xp.n_total + my_env) * 2;
          rec[0] = (uint8_t)act0;
          rec[1] = (uint8_t)act1;
        }
        float r0, r1, team;
        const int done = Env::step(a.b.env, s2, act0, act1, r0, r1, team);
        if (done < 0) {
          atomicOr(a.b.status, kStatusIllegalAction);
          alive = false;
        } else {
          nsteps += 1;
          if (done) alive = false;
        }
        st[row] = s2;
      } else if (!kXp && ag == 0 && half == 0 && row < count) {
        State s2 = s;
        const int act1 = act1s[row];
        const int64_t env = my_env;
        if constexpr (kGather) {
          if (a.g.teammate) a.g.teammate[env] = tm_pol;
          if (a.g.teammate2) a.g.teammate2[env] = tm_pol;
        }
        float r0, r1, team;
        const int done = Env::step(a.b.env, s2, act0, act1, r0, r1, team);
        const int64_t o = (int64_t)t * N + env;
        if (a.traj.actions) a.traj.actions[o] = (uint8_t)act0;
        if (a.traj.tm_actions) a.traj.tm_actions[o] = (uint8_t)act1;
        if (a.traj.logp) a.traj.logp[o] = lp0;
        if (a.traj.values) a.traj.values[o] = val0;
        if (a.traj.rewards) a.traj.rewards[o] = team;
        if (a.traj.dones) a.traj.dones[o] = (uint8_t)(done > 0);
        if constexpr (kIppo) {  // seat 1's learner fields
          if (a.traj1.actions) a.traj1.actions[o] = (uint8_t)act1;
          if (a.traj1.tm_actions) a.traj1.tm_actions[o] = (uint8_t)act0;
          if (a.traj1.rewards) a.traj1.rewards[o] = team;
          if (a.traj1.dones) a.traj1.dones[o] = (uint8_t)(done > 0);
        }
        if (done > 0) {
          Env::reset(a.b.env, a.b.key, (uint32_t)env, gt + 1, s2);
          if (a.ep_step) a.ep_step[env] = gt + 1;
        }
        if (kGather && a.g.resample) {  // the next step's pool index: a new episode draws again
          int kn = g_k;
          if (done > 0) {
            kn = (int)uniform_int(draw0(a.b.key, (uint32_t)env, gt + 1, kStreamEpisodeTeammate),
                                  (uint32_t)a.g.pool_size);
            atomicAdd(&a.g.hist_next[kn], 1);
          }
          a.g.kidx_next[env] = (uint8_t)kn;
          stayed = done <= 0;
        }
        st[row] = s2;
      }
      if (kGather && a.g.resample && ag == 0 && half == 0) {
        const unsigned m = __ballot_sync(0xFFFFFFFFu, stayed);
        if (lane == 0 && m) atomicAdd(&a.g.hist_next[g_k], __popc(m));
      }
      if (obs_copy && (ag == 1 || half == 1)) copy_rows_gathered(t, ag == 1 ? warp - 8 : warp + 4);
      if (kIppo && a.traj1.obs && (ag == 1 || half == 1)) {  // seat 1's rows, a contiguous block
        const int cw = ag == 1 ? warp - 8 : warp + 4;
        const uint32_t* const src = reinterpret_cast<const uint32_t*>(sObs);
        uint32_t* const dst = reinterpret_cast<uint32_t*>(a.traj1.obs + ((int64_t)t * N + env0) * od);
        for (int f = cw * 32 + lane; f < count * cells; f += 12 * 32) dst[f] = Env::other_seat_word(src[f]);
      }
      if (tid == 0 && bulk_obs) tc::bulk_wait_read();  // the rows may be rebuilt
      if (sync_all()) break;                            // the new state is in place
    }
    if (tid == 0 && bulk_obs) tc::bulk_wait_all();
    if (bad) {
      atomicOr(a.b.status, kStatusTimeout);
      // cross-play: the tile gave up, so its returns are undefined; NaN (not a stale entry
      // of an earlier call) makes every mean over them NaN
      if (kXp && tid < count) a.xp.returns[env0 + tid] = __int_as_float(0x7FC00000);
    } else if (tid < count) {
      if constexpr (kXp) {
        a.xp.returns[env0 + tid] = Env::ret(st[tid]);
      } else {
        store_state(a.state, N, env_of(tid), st[tid]);
      }
    }
    if (kXp && a.xp.steps && !bad && ag == 0 && half == 0 && row < count) a.xp.steps[env0 + row] = nsteps;
    // ---- drain: every MMA this thread issued completes (bounded) ----
    if (leader && n_issued > 0) {
      tc::commit(&drain_bar[ag]);
      tc::mbar_wait(&drain_bar[ag], 0);
    }
  }

  // ---- then free tensor memory ----
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 0) {
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, 512);
  }
}

template <class Env>
struct LaunchTc2 {
  template <bool kSplit, bool kGather, bool kXp = false, bool kIppo = false>
  static cudaError_t run(const PpoTcArgs& a, int grid, size_t smem, cudaStream_t s) {
    cudaError_t e = cudaFuncSetAttribute(ppo2_tc_kernel<Env, kSplit, kGather, kXp, kIppo>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)grid);
    cfg.blockDim = dim3(kT2Threads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = a.pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, ppo2_tc_kernel<Env, kSplit, kGather, kXp, kIppo>, a);
  }
  // IPPO collection (dense first layer, contiguous tiles)
  static cudaError_t ippo(const PpoTcArgs& a, int grid, size_t smem, cudaStream_t s) {
    return a.tc.split ? run<true, false, false, true>(a, grid, smem, s) : run<false, false, false, true>(a, grid, smem, s);
  }
  // cross-play (dense first layer)
  static cudaError_t xplay(const PpoTcArgs& a, int grid, size_t smem, cudaStream_t s) {
    return a.tc.split ? run<true, false, true>(a, grid, smem, s) : run<false, false, true>(a, grid, smem, s);
  }
  // plain PPO collection (no IPPO, dense first layer)
  static cudaError_t ppo(const PpoTcArgs& a, int grid, size_t smem, cudaStream_t s) {
    if (a.gather) return a.tc.split ? run<true, true>(a, grid, smem, s) : run<false, true>(a, grid, smem, s);
    return a.tc.split ? run<true, false>(a, grid, smem, s) : run<false, false>(a, grid, smem, s);
  }
};

}  // namespace aht
