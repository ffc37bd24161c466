// rollout_tc.cuh -- fused LBF rollout with a sparse first layer and the rest of the policy
// MLPs on tcgen05 tensor cores.
//
// The kernel serves LBF observations wider than the 256 tensor-memory columns of an
// agent's A operand (the 12x12 grid's 576 features): PPO collection (a contiguous env
// range for a one-member pool, else the envs of one teammate's group found by a rank
// scan of the per-env pool indices, kGather) and cross-play (kXp).  Every LBF launch with
// a dense first layer runs on the two-group kernel of rollout_tc2.cuh, which shares this
// file's tile finder.  One CTA owns a tile of up to 128 envs that share one teammate
// policy, for all T steps.  Per step and agent (teammate first, then the ego = seat 0):
//   h1 on CUDA cores: the observation is a fixed pattern plus at most ten changed
//       features, so r1 = 1 / (1 + exp(2 (c + sum over them of delta W1[:, f]))), c = b1 +
//       W1 x_pattern; r1 is split r1 = hi + lo (two bf16) into tensor memory.  tanh(x) =
//       1 - 2 r1, and the block's W2, b2 hold -2 W2 and b2 + W2 1, so L2 sees exactly the
//       tanh layer (the same for r2 and W3, b3 below)
//   L2 (tensor cores): D = hi W2'^T + lo W2'^T  (the split keeps ~2^-17 relative precision
//       of r1 with bf16 operands and fp32 accumulate)
//   epilogue 2: r2 = 1 / (1 + exp(2 (D + b2))), split again, and z = W3' r2 + b3' by mma.sync m16n8k16
//       from registers (16x256b accumulator loads are its fragment layout)
//   sampling (ego in warps 0-3, teammate in warps 4-7), env step, trajectory write.
//
// Warp roles: warps 0-7 ("compute", 256 threads) build the ego's observation rows for the
// trajectory, form h1, run epilogue 2 (thread r and r + 128 own env row r, tensor-memory
// lane r; the halves split the columns), sample and step the envs; warp 8 issues every
// MMA; warps 9-12 store the ego's observation rows of gathered tiles (scattered rows, a
// quarter each, one warp per SM sub-partition) while the compute warps go on.  They meet
// only through mbarriers: operand-ready (256 arrivals from the compute threads) and
// accumulator-ready (a tcgen05.commit); observation rows ready (256 arrivals) and
// observation buffer free (one arrival per store warp).  Each of these barriers completes
// once per step, so its phase parity is the step's parity.  Compute warps synchronise
// among themselves with a named barrier that also ORs an error flag.  Weights (all but
// W1) are bulk-copied (TMA) into shared memory once per CTA; W1^T and c are read from
// the L2-resident fp32 population.  Every wait is bounded: on expiry the CTA records
// kStatusTimeout, stops, drains its own MMAs (bounded), frees tensor memory and exits.
//
// Tensor memory (512 columns): agent a uses columns [256a, 256a + 128) for its A operand
// (hi|lo of h1) and [256a + 128, 256a + 256) for its fp32 accumulator.
#pragma once
#include "kernels.h"
#include "rollout_impl.cuh"
#include "tc_common.cuh"

namespace aht {

constexpr int kTcCompute = 256;          // compute threads
constexpr int kTcThreads = 416;          // + one MMA warp + four observation-store warps
constexpr int kTcStoreWarps = 4;         // warps 9-12: one per SM sub-partition
constexpr int kTcComputeBar = 1;         // named barrier id of the compute warps

// The tile of CTA blockIdx.x: cross-play (kXp) chunk `blockIdx.x % tpp` of pair
// `blockIdx.x / tpp`; gathered (kGather) tile blockIdx.x of the teammate groups, its envs
// found by a rank scan of the per-env pool indices into rowenv[0 .. count); otherwise
// entry blockIdx.x of the contiguous tile table.  Every thread of the block calls it (it
// synchronises the block); blockDim.x <= 24 warps.
struct TcTile {
  int64_t env0;   // first env (contiguous tiles)
  int count;      // rows (0: nothing to do)
  int ego_pol, tm_pol;
  int g_k;        // gathered: the tile's pool index
};
template <bool kXp, bool kGather>
__device__ __forceinline__ TcTile tc_find_tile(const PpoTcArgs& a, int32_t* rowenv) {
  int64_t env0;
  int count, ego_pol, tm_pol;
  int g_k = 0;                                      // gather: the tile's pool index
  if constexpr (kXp) {
    const int pair = blockIdx.x / a.xp.tpp, chunk = blockIdx.x - pair * a.xp.tpp;
    env0 = (int64_t)pair * a.xp.P + 128 * chunk;
    count = min(128, a.xp.P - 128 * chunk);
    ego_pol = a.xp.ego_ids[pair / a.xp.n_tm];
    tm_pol = a.xp.tm_ids[pair % a.xp.n_tm];
  } else if constexpr (kGather) {
    // Tile blockIdx.x of the groups in pool-index order: group k holds hist_cur[k] envs,
    // cut into tiles of up to M in env order.  Rows are found by a rank scan of kidx:
    // each thread counts its contiguous chunk's envs of group k, an exclusive scan gives
    // the chunk's first rank, and the envs of ranks [r0, r0 + count) become rows.
    int* wsum = reinterpret_cast<int*>(rowenv + 128);  // [0, 24) warp totals, [28, 31) selection
    const int t0 = threadIdx.x, w0 = t0 >> 5, l0 = t0 & 31;
    if (blockIdx.x == 0 && a.g.resample)
      for (int k = t0; k < a.g.pool_size; k += blockDim.x) a.g.hist_zero[k] = 0;
    if (t0 < 128) rowenv[t0] = -1;
    if (t0 == 0) {
      const int M = a.g.M;
      int cum = 0, ks = -1, r0 = 0, cnt = 0;
      for (int k = 0; k < a.g.pool_size; ++k) {
        const int h = a.g.hist_cur[k], nt = (h + M - 1) / M;
        if (ks < 0 && (int)blockIdx.x < cum + nt) {
          ks = k;
          r0 = ((int)blockIdx.x - cum) * M;
          cnt = min(M, h - r0);
        }
        cum += nt;
      }
      wsum[28] = ks;
      wsum[29] = r0;
      wsum[30] = ks < 0 ? 0 : cnt;
    }
    __syncthreads();
    g_k = wsum[28];
    const int r0 = wsum[29];
    count = wsum[30];
    env0 = 0;
    ego_pol = a.ego;
    tm_pol = g_k < 0 ? 0 : a.g.pool[g_k];
    if (count > 0) {  // block-uniform
      const int64_t n = a.n_envs, nthr = blockDim.x;
      const int64_t C = (((n + nthr - 1) / nthr) + 15) & ~(int64_t)15;  // bytes per thread
      const int64_t b0 = t0 * C, b1 = min(n, b0 + C);
      const uint8_t* kx = a.g.kidx_cur;
      const uint32_t kk = 0x01010101u * (uint32_t)g_k;
      // 16 indices of [e, e + 16) as match bytes (0xFF where kidx == g_k, 0 past b1);
      // b0 is a multiple of 16 and kidx is 16-byte aligned
      auto matches = [&](int64_t e) {
        uint4 m;
        if (e + 16 <= b1) {
          const uint4 v = __ldg(reinterpret_cast<const uint4*>(kx + e));
          m = make_uint4(__vcmpeq4(v.x, kk), __vcmpeq4(v.y, kk), __vcmpeq4(v.z, kk), __vcmpeq4(v.w, kk));
        } else {
          uint32_t w[4] = {0u, 0u, 0u, 0u};
          for (int64_t f = e; f < b1; ++f)
            if (kx[f] == (uint8_t)g_k) w[(f - e) >> 2] |= 0xFFu << (8 * ((f - e) & 3));
          m = make_uint4(w[0], w[1], w[2], w[3]);
        }
        return m;
      };
      int c = 0;
#pragma unroll 4
      for (int64_t e = b0; e < b1; e += 16) {
        const uint4 m = matches(e);
        c += (__popc(m.x) + __popc(m.y) + __popc(m.z) + __popc(m.w)) >> 3;
      }
      int incl = c;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
        if (l0 >= o) incl += y;
      }
      if (l0 == 31) wsum[w0] = incl;
      __syncthreads();
      int rank = incl - c;
      for (int w = 0; w < w0; ++w) rank += wsum[w];
      if (c > 0 && rank < r0 + count && rank + c > r0) {
#pragma unroll 4
        for (int64_t e = b0; e < b1; e += 16) {
          const uint4 m = matches(e);
          const uint32_t mw[4] = {m.x, m.y, m.z, m.w};
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            uint32_t bits = mw[q] & 0x80808080u;  // one bit per matching byte
            while (bits) {
              const int byte = (__ffs(bits) - 1) >> 3;
              bits &= bits - 1;
              if (rank >= r0 && rank < r0 + count) rowenv[rank - r0] = (int32_t)(e + 4 * q + byte);
              ++rank;
            }
          }
        }
      }
    }
    __syncthreads();
    // every row must have found its env (the counts and the indices agree by
    // construction); otherwise the tile is skipped and the status word says so
    if (!__syncthreads_and(t0 >= count || (rowenv[t0] >= 0 && rowenv[t0] < a.n_envs))) {
      if (t0 == 0) atomicOr(a.b.status, kStatusGrouping);
      count = 0;
    }
  } else {
    const int4 tile = a.tiles[blockIdx.x];
    env0 = tile.x;
    count = tile.y;
    ego_pol = a.ego;
    tm_pol = tile.z;
  }
  return TcTile{env0, count, ego_pol, tm_pol, g_k};
}

// kXp: cross-play (each tile is a chunk of one pair's envs, reset at the call's first
// step, frozen once done; the per-env return and episode length are the outputs) instead
// of PPO collection.  kSplit: fp32 weights held as bf16 pairs W = W_hi + W_lo and L2 = b2
// + hi W2_hi + lo W2_hi + hi W2_lo (lo W2_lo is below 2^-16 of the sum and left out).
// kGather (PPO collection): the tile's rows are envs of one teammate group found by a rank
// scan of the per-env pool indices (the call's draw, held for all T steps) instead of a
// contiguous range.  Env::sparse_obs lists the changed features; W1^T and c are the fp32
// copies of the CUDA-core population.
template <class Env, bool kXp, bool kSplit, bool kGather>
__global__ void __launch_bounds__(kTcThreads, 1) ppo_tc_kernel(const PpoTcArgs a) {
  static_assert(!(kGather && kXp), "gathered tiles are PPO collection");
  static_assert(kTcThreads / 32 <= 24, "gather scratch: one total per warp");
  using State = typename Env::State;
  constexpr int NA = Env::kNumActions;
  extern __shared__ __align__(16) uint8_t smem[];  // no-swizzle operands need 16 B
  __shared__ __align__(8) uint64_t acc_bar[2];     // [agent], L2 committed (tcgen05.commit)
  __shared__ __align__(8) uint64_t opnd_bar[2];    // [agent], h1 in tensor memory (256 arrivals)
  __shared__ __align__(8) uint64_t wload_bar, drain_bar;
  __shared__ __align__(8) uint64_t obs_full, obs_free;  // gathered observation rows: warps 9-12
  __shared__ __align__(8) uint64_t never_bar;           // test hook: nothing arrives on it
  __shared__ uint32_t tmem_slot;
  __shared__ volatile int abort_flag;
  __shared__ volatile int stop_flag;               // cross-play: every env of the tile is done

  int32_t* const rowenv = kGather ? reinterpret_cast<int32_t*>(smem + a.g.scratch_off) : nullptr;
  const TcTile tile = tc_find_tile<kXp, kGather>(a, rowenv);
  const int64_t env0 = tile.env0;
  const int count = tile.count, ego_pol = tile.ego_pol, tm_pol = tile.tm_pol;
  if (count <= 0) return;
  // a negative teammate id is LBF heuristic -1 - id: no teammate network, its rule acts
  const bool tm_rule = tm_pol < 0;
  const TcDims& d = a.tc;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, half = (warp >> 2) & 1, row = tid & 127;
  // env index of tile row r (r < count)
  auto env_of = [&](int r) -> int64_t { return kGather ? (int64_t)rowenv[r] : env0 + r; };
  const int64_t my_env = row < count ? env_of(row) : 0;
  const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;
  const int64_t N = a.n_envs;
  const int od = a.b.env.obs_dim;
  const int cells = od / 4;          // observation words per row
  const int chunks = d.KP / 16;      // 16-byte chunks per observation row
  const int split = (chunks + 1) / 2;
  // the halves build words [my_w0, my_w1) of the ego's row
  const int my_w0 = min(4 * (half ? split : 0), cells), my_w1 = min(4 * (half ? chunks : split), cells);
  const bool with_boot = !kXp && a.traj.last_value != nullptr;  // the ego's V_T after the last step
  // gathered tiles: warps 9-12 store the ego's observation rows of every step
  const bool obs_warp = kGather && a.traj.obs != nullptr;

  // The tile is the contiguous env range [tile.x, tile.x + count); observation rows are
  // packed at obs_dim bytes (an odd number of words: no bank conflicts per thread row),
  // so the tile's rows form one contiguous block for a single bulk store.
  uint8_t* const sW0 = smem;                                                // policy blocks
  uint8_t* const sObs = smem + 2 * d.pol_bytes;                             // [128][obs_dim] u8
  State* st = reinterpret_cast<State*>(sObs + align_up(128 * od, 16));      // [128]
  uint8_t* act1s = reinterpret_cast<uint8_t*>(st) + align_up(128 * sizeof(State), 16);  // [128]
  float* zpart = reinterpret_cast<float*>(act1s + 128);                     // [2][2][128][8]

  if (tid == 0) {
    for (int i = 0; i < 2; ++i) {
      tc::mbar_init(&acc_bar[i], 1);
      tc::mbar_init(&opnd_bar[i], kTcCompute);
    }
    tc::mbar_init(&wload_bar, 1);
    tc::mbar_init(&drain_bar, 1);
    tc::mbar_init(&obs_full, kTcCompute);
    tc::mbar_init(&obs_free, kTcStoreWarps);
    tc::mbar_init(&never_bar, 1);
    tc::mbar_init_fence();
    abort_flag = 0;
    stop_flag = 0;
  }
  if (warp == 0) tc::tmem_alloc(&tmem_slot, 512);
  for (int i = tid; i < 32 * od; i += blockDim.x) reinterpret_cast<uint32_t*>(sObs)[i] = 0u;
  if (tid < count) {
    if constexpr (kXp) Env::reset(a.b.env, a.b.key, (uint32_t)(env0 + tid), a.step0, st[tid]);
    else load_state(a.state, N, env_of(tid), st[tid]);
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = tmem_slot;

  if (warp == 8) {
    // ================================ MMA warp =====================================
    if (lane == 0) {
      const int pol[2] = {ego_pol, tm_pol};
      const int n_pol = tm_rule ? 1 : 2;
      tc::mbar_expect_tx(&wload_bar, (uint32_t)n_pol * d.pol_bytes);
      for (int p = 0; p < n_pol; ++p) {
        const uint8_t* src = a.tcw + (int64_t)pol[p] * d.pol_bytes;
        for (uint32_t off = 0; off < d.pol_bytes; off += 32768u)
          tc::bulk_g2s(sW0 + p * d.pol_bytes + off, src + off, min(32768u, d.pol_bytes - off), &wload_bar);
      }
      bool ok = tc::mbar_wait(&wload_bar, 0);
      const uint32_t idesc2 = tc::idesc_bf16(128, d.H1);
      const uint32_t sbo2 = (uint32_t)(d.H0 / 8) * 128u;
      // agents in the order the compute warps release them: teammate, then ego
      bool stopped = false;
      auto issue = [&](int ag, uint32_t parity) {  // L2 of agent ag
        ok = false;
        for (int tries = 0; tries < 1000 && !ok && !abort_flag; ++tries)
          ok = tc::mbar_wait(&opnd_bar[ag], parity, 2000000ull);
        if (!ok) return;
        if (kXp && stop_flag) {  // released without operands: the tile is finished
          stopped = true;
          return;
        }
        tc::fence_after_sync();
        const uint32_t wbase = tc::smem_u32(sW0) + (uint32_t)ag * d.pol_bytes;
        const uint32_t P = tmem + (uint32_t)(ag * 256), Q = P + 128;
        const uint64_t w0 = tc::smem_desc(wbase + d.oW2, 128u, sbo2);
        for (int ks = 0; ks < d.H0 / 16; ++ks) tc::mma_ts(Q, P + 8 * ks, w0 + 16u * ks, idesc2, ks > 0);
        for (int ks = 0; ks < d.H0 / 16; ++ks) tc::mma_ts(Q, P + d.H0 / 2 + 8 * ks, w0 + 16u * ks, idesc2, 1u);
        if constexpr (kSplit) {
          const uint64_t w1 = tc::smem_desc(wbase + d.oW2lo, 128u, sbo2);
          for (int ks = 0; ks < d.H0 / 16; ++ks) tc::mma_ts(Q, P + 8 * ks, w1 + 16u * ks, idesc2, 1u);
        }
        tc::commit(&acc_bar[ag]);
      };
      const int n_steps = kXp ? a.xp.max_steps : a.T;
      for (int t = 0; ok && !stopped && t < n_steps; ++t) {
        const uint32_t par = (uint32_t)t & 1u;
        if (!tm_rule) issue(1, par);
        if (ok && !stopped) issue(0, par);
      }
      if (ok && with_boot) issue(0, (uint32_t)a.T & 1u);
      if (!ok) abort_flag = 1;
    }
  } else if (warp > 8) {
    // ======================= observation-store warps (gathered) =====================
    // Step t's ego rows (built by the compute warps, obs_full phase t) go to their envs'
    // trajectory rows with consecutive words, warp 9 + q taking rows q, q + 4, ...;
    // obs_free (one arrival per warp) tells the compute warps that the buffer may be
    // rebuilt.
    const int q = warp - 9;
    for (int t = 0; obs_warp && t < a.T; ++t) {
      int ok = 0;
      if (lane == 0)
        for (int tries = 0; tries < 1000 && !ok && !abort_flag; ++tries)
          ok = tc::mbar_wait(&obs_full, (uint32_t)t & 1u, 2000000ull);
      ok = __shfl_sync(0xFFFFFFFFu, ok, 0);
      __syncwarp();
      if (!ok) break;  // the compute warps gave up
      // lane l moves word w0 + l of 8 rows per iteration: 8 independent shared-memory
      // loads in flight, then 8 stores (each row's words leave as consecutive words)
      uint32_t* const base = reinterpret_cast<uint32_t*>(a.traj.obs + (int64_t)t * N * od);
      const uint32_t* const src = reinterpret_cast<const uint32_t*>(sObs);
      for (int w0 = 0; w0 < cells; w0 += 32) {
        const int w = w0 + lane;
        const bool wok = w < cells;
#pragma unroll 1
        for (int r0 = q; r0 < count; r0 += 4 * 8) {
          uint32_t v[8];
          int64_t dst[8];
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const int r = min(r0 + 4 * j, count - 1);
            dst[j] = (int64_t)rowenv[r] * cells + w;
            v[j] = wok ? src[r * cells + w] : 0u;
          }
#pragma unroll
          for (int j = 0; j < 8; ++j)
            if (wok && r0 + 4 * j < count) base[dst[j]] = v[j];
        }
      }
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&obs_free);
    }
  } else {
    // ============================== compute warps ===================================
    bool bad = false;
    auto wait_acc = [&](int ag, uint32_t parity) {
      if (!bad && !tc::mbar_wait(&acc_bar[ag], parity)) bad = true;
      bad = __any_sync(0xFFFFFFFFu, bad);  // warp-uniform: tensor-memory loads are collective
      tc::fence_after_sync();
    };
    auto operand_ready = [&](int ag) {  // this thread's tensor-memory traffic is done
      tc::fence_before_sync();
      tc::mbar_arrive(&opnd_bar[ag]);
    };
    auto sync_or = [&]() { return tc::bar_or(kTcComputeBar, kTcCompute, bad || abort_flag); };
    auto pol_block = [&](int ag) { return sW0 + (size_t)ag * d.pol_bytes; };

    // h1: r1 = 1 / (1 + exp(2 (c + sum over the changed features f of delta W1[:, f]))) for this
    // thread's half of the units, split hi | lo into the A operand of L2; rows past count
    // take c alone.  The W1 rows are gathered 8 units at a time with all ten
    // features' loads issued before their multiply-adds (one L2 round trip per 8 units,
    // not one per feature); an absent feature reads row 0 and adds 0 x W1 (exact)
    auto sparse_h1 = [&](int ag, const State& s) {
      const int H = d.H0;
      const uint32_t P = tmem + (uint32_t)(ag * 256) + lane_base;
      const float* pw = a.b.weights + (int64_t)(ag == 0 ? ego_pol : tm_pol) * a.b.mlp.stride;
      const float* W1t = pw + a.b.mlp.oW1;
      const float* cvec = pw + a.b.mlp.oC;
      uint32_t e[10];
      const uint32_t mask = row < count ? Env::sparse_obs(a.b.env, s, ag, e) : 0u;
#pragma unroll 1
      for (int c0 = half * (H / 2); c0 < (half + 1) * (H / 2); c0 += 16) {
        float v[16];
#pragma unroll
        for (int j = 0; j < 16; j += 4) {
          const float4 cc = __ldg(reinterpret_cast<const float4*>(cvec + c0 + j));
          v[j] = cc.x; v[j + 1] = cc.y; v[j + 2] = cc.z; v[j + 3] = cc.w;
        }
#pragma unroll
        for (int j8 = 0; j8 < 16; j8 += 8) {
          float4 w4[10][2];
#pragma unroll
          for (int q = 0; q < 10; ++q) {
            const uint32_t f = (mask >> q) & 1u ? e[q] >> 8 : 0u;
            const float* wr = W1t + (int64_t)f * H + c0 + j8;
            w4[q][0] = __ldg(reinterpret_cast<const float4*>(wr));
            w4[q][1] = __ldg(reinterpret_cast<const float4*>(wr + 4));
          }
#pragma unroll
          for (int q = 0; q < 10; ++q) {
            const float dv = (mask >> q) & 1u ? (float)(int8_t)(e[q] & 0xFFu) : 0.0f;
#pragma unroll
            for (int k = 0; k < 2; ++k) {
              float* vv = v + j8 + 4 * k;
              vv[0] = fmaf(dv, w4[q][k].x, vv[0]);
              vv[1] = fmaf(dv, w4[q][k].y, vv[1]);
              vv[2] = fmaf(dv, w4[q][k].z, vv[2]);
              vv[3] = fmaf(dv, w4[q][k].w, vv[3]);
            }
          }
        }
        uint32_t hi[8], lo[8];
#pragma unroll
        for (int j = 0; j < 8; ++j)
          tc::split_bf16x2_p(tc::logistic2(tc::f2_mul(tc::f2_pack(v[2 * j], v[2 * j + 1]), tc::kTwoOverLn2x2)), hi[j], lo[j]);
        tc::st_x8(P + c0 / 2, hi);
        tc::st_x8(P + H / 2 + c0 / 2, lo);
      }
      tc::wait_st();
      operand_ready(ag);
    };
    // epilogue 2: r2 = 1 / (1 + exp(2 (D + b2))) and this half's partial z = sum_k W3'[:, k] r2[k] on the
    // tensor cores from registers (mma.sync m16n8k16, one n-tile of 8 outputs): the warp
    // takes its 32 rows as two groups of 16 and its half's units as chunks of 16; two
    // 16x256b loads of the accumulator give the thread its A fragment (rows g, g + 8 with
    // g = lane / 4; units 2c, 2c + 1 and 2c + 8, 2c + 9 of the chunk, c = lane % 4);
    // r2 = hi + lo (two bf16) and z += hi W3'^T + lo W3'^T (+ hi W3lo'^T for
    // split blocks), fp32 accumulate.  The partial sums go to shared memory for the
    // sampling half.
    auto epilogue2 = [&](int ag) {
      const int H = d.H1;
      const float* b2 = reinterpret_cast<const float*>(pol_block(ag) + d.ob2);
      const uint32_t Qq = tmem + (uint32_t)(ag * 256 + 128) + ((uint32_t)((warp & 3) * 32) << 16);
      const uint32_t* W3f = reinterpret_cast<const uint32_t*>(pol_block(ag) + d.oW3);
      const uint32_t* W3l = W3f + H * 4;  // split blocks: the remainders
      const int g = lane >> 2, c4 = lane & 3;
      float zacc[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
#pragma unroll 1
      for (int c0 = half * (H / 2); c0 < (half + 1) * (H / 2); c0 += 16) {
        const int j = c0 >> 4;
        const uint2 bw = *reinterpret_cast<const uint2*>(W3f + (j * 32 + lane) * 2);
        const uint64_t bA = *reinterpret_cast<const uint64_t*>(b2 + c0 + 2 * c4);
        const uint64_t bB = *reinterpret_cast<const uint64_t*>(b2 + c0 + 8 + 2 * c4);
        uint2 bl = make_uint2(0u, 0u);
        if constexpr (kSplit) bl = *reinterpret_cast<const uint2*>(W3l + (j * 32 + lane) * 2);
#pragma unroll
        for (int rg = 0; rg < 2; ++rg) {
          uint32_t t0[4], t1[4];
          tc::ld_16x256b(Qq + ((uint32_t)(16 * rg) << 16) + (uint32_t)c0, t0);
          tc::ld_16x256b(Qq + ((uint32_t)(16 * rg) << 16) + (uint32_t)(c0 + 8), t1);
          tc::wait_ld();
          uint32_t ahi[4], alo[4];
          tc::split_bf16x2_p(tc::logistic2(tc::f2_fma(tc::f2_pack(__uint_as_float(t0[0]), __uint_as_float(t0[1])), tc::kTwoOverLn2x2, bA)),
                             ahi[0], alo[0]);
          tc::split_bf16x2_p(tc::logistic2(tc::f2_fma(tc::f2_pack(__uint_as_float(t0[2]), __uint_as_float(t0[3])), tc::kTwoOverLn2x2, bA)),
                             ahi[1], alo[1]);
          tc::split_bf16x2_p(tc::logistic2(tc::f2_fma(tc::f2_pack(__uint_as_float(t1[0]), __uint_as_float(t1[1])), tc::kTwoOverLn2x2, bB)),
                             ahi[2], alo[2]);
          tc::split_bf16x2_p(tc::logistic2(tc::f2_fma(tc::f2_pack(__uint_as_float(t1[2]), __uint_as_float(t1[3])), tc::kTwoOverLn2x2, bB)),
                             ahi[3], alo[3]);
          tc::mma_m16n8k16_bf16(zacc[rg], ahi, bw.x, bw.y);
          tc::mma_m16n8k16_bf16(zacc[rg], alo, bw.x, bw.y);
          if constexpr (kSplit) tc::mma_m16n8k16_bf16(zacc[rg], ahi, bl.x, bl.y);
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
    // full logits of agent ag: (half-0 partial + half-1 partial) + b3
    auto logits = [&](int ag, float (&z)[16]) {
      const float* p0 = zpart + ((ag * 2 + 0) * 128 + row) * 8;
      const float* p1 = zpart + ((ag * 2 + 1) * 128 + row) * 8;
      const float* b3 = reinterpret_cast<const float*>(pol_block(ag) + d.ob3);
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
    // the tile's ego observation rows -> trajectory [t][env0 .. env0+count): one contiguous
    // block, written by one bulk (TMA) store when 16-byte aligned, else by all threads
    // (gathered tiles: warp 9)
    const bool bulk_obs = !kXp && !kGather && a.traj.obs && (count * od) % 16 == 0;
    auto copy_obs = [&](int t) {
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
        for (uint32_t w = tid; w < bytes / 4; w += kTcCompute) d32[w] = src[w];
      }
    };

    // Steps 0..T-1, then (if requested) the ego's V_T of the state after the last step.
    // The agent loops are not unrolled so that every phase's code exists once.
    const int n_steps = kXp ? a.xp.max_steps : a.T;
    bool alive = true;  // cross-play: the row's episode is running (half-0 threads)
    int nsteps = 0;
    for (int t = 0; t <= n_steps; ++t) {
      const bool boot = t == n_steps;
      if (boot && !with_boot) break;
      if constexpr (kXp) {
        // every env of the tile is done: release the MMA warp without operands and stop
        if (!tc::bar_or(kTcComputeBar, kTcCompute, half == 0 && row < count && alive)) {
          if (tid == 0) stop_flag = 1;
          tc::mbar_arrive(&opnd_bar[tm_rule ? 0 : 1]);  // the first barrier it waits on
          break;
        }
      }
      // gathered tiles: the previous step's ego rows must have left the buffer
      if (obs_warp && t >= 1) {
        if (!bad && !tc::mbar_wait(&obs_free, (uint32_t)(t - 1) & 1u)) bad = true;
        bad = __any_sync(0xFFFFFFFFu, bad);
      }
      // teammate first (its network runs in every step but the bootstrap)
      const int first = boot || tm_rule ? 0 : 1;
      const uint32_t par = (uint32_t)t & 1u, gt = a.step0 + (uint32_t)t;
      // this half's action draw (ego: warps 0-3, teammate: warps 4-7), ahead of its use
      const float u_act = boot ? 0.0f : u01(draw0(a.b.key, (uint32_t)my_env, gt, kStreamAct0 + half));
      State s = st[row];  // register copy for this step (rows past count are never used)
#pragma unroll 1
      for (int i = first; i >= 0; --i) {
        // the ego's u8 row is the trajectory's observation; no first layer to feed
        if (!kXp && i == 0 && !boot && a.traj.obs && row < count)
          Env::obs_words(a.b.env, s, 0, reinterpret_cast<uint32_t*>(sObs + row * od), my_w0, my_w1);
        if (obs_warp && i == 0 && !boot) tc::mbar_arrive(&obs_full);
        if (!bad) sparse_h1(i, s);
      }
      if (t == a.dbg_expire_step) {  // test hook: an accumulator wait that never completes
        if (!bad && !tc::mbar_wait(&never_bar, 0, a.dbg_expire_ns)) bad = true;
        bad = __any_sync(0xFFFFFFFFu, bad);
      }
      if (!kXp && !kGather && !boot && a.traj.obs) {  // overlaps L2 on the tensor cores
        tc::fence_proxy_async();       // the rows were written by ordinary stores
        if (sync_or()) break;
        copy_obs(t);
      }
#pragma unroll 1
      for (int i = first; i >= 0; --i) {
        wait_acc(i, par);
        if (!bad) epilogue2(i);
      }
      if (sync_or()) break;
      float z[16];
      if (boot) {
        if (half == 0 && row < count) {
          logits(0, z);
          a.traj.last_value[my_env] = z[NA];
        }
        break;
      }
      int act0 = 0;
      float lp0 = 0.f, val0 = 0.f;
      if (row < count && half == 1 && tm_rule) {
        act1s[row] = (uint8_t)Env::heuristic(a.b.env, st[row], -1 - tm_pol);  // st[row] == s here
      } else if (row < count) {
        const int ag = half == 0 ? 0 : 1;
        logits(ag, z);
        if (a.dbg_logits) {  // test hook: this row's outputs of step t (frozen rows too)
          const int64_t rows = kXp ? a.xp.n_total : N;
          float* p = a.dbg_logits + (((int64_t)t * rows + my_env) * 2 + ag) * kDbgStride;
#pragma unroll
          for (int o = 0; o < 8; ++o) p[o] = z[o];
        }
        float lp;
        const int act = sample_k<NA>(z, 0xFFFFFFFFu >> (32 - NA), u_act, lp);
        if (ag == 1) {
          act1s[row] = (uint8_t)act;
        } else {
          act0 = act;
          lp0 = lp;
          val0 = z[NA];
        }
      }
      if (sync_or()) break;
      if (kXp && half == 0 && row < count && alive) {
        const int act1 = act1s[row];
        const int64_t env = env0 + row;
        if (a.xp.actions) {
          uint8_t* rec = a.xp.actions + ((int64_t)t * a.xp.n_total + env) * 2;
          rec[0] = (uint8_t)act0;
          rec[1] = (uint8_t)act1;
        }
        float r0, r1, team;
        const int done = Env::step(a.b.env, s, act0, act1, r0, r1, team);
        if (done < 0) {
          atomicOr(a.b.status, kStatusIllegalAction);
          alive = false;
        } else {
          nsteps += 1;
          if (done) alive = false;
        }
        st[row] = s;
      } else if (!kXp && half == 0 && row < count) {
        const int act1 = act1s[row];
        const int64_t env = my_env;
        if constexpr (kGather) {
          if (a.g.teammate) a.g.teammate[env] = tm_pol;
          if (a.g.teammate2) a.g.teammate2[env] = tm_pol;
        }
        float r0, r1, team;
        const int done = Env::step(a.b.env, s, act0, act1, r0, r1, team);
        const int64_t o = (int64_t)t * N + env;
        if (a.traj.actions) a.traj.actions[o] = (uint8_t)act0;
        if (a.traj.tm_actions) a.traj.tm_actions[o] = (uint8_t)act1;
        if (a.traj.logp) a.traj.logp[o] = lp0;
        if (a.traj.values) a.traj.values[o] = val0;
        if (a.traj.rewards) a.traj.rewards[o] = team;
        if (a.traj.dones) a.traj.dones[o] = (uint8_t)(done > 0);
        if (done > 0) {
          Env::reset(a.b.env, a.b.key, (uint32_t)env, gt + 1, s);
          if (a.ep_step) a.ep_step[env] = gt + 1;
        }
        st[row] = s;
      }
      if (tid == 0 && bulk_obs) tc::bulk_wait_read();  // the rows may be rebuilt
      if (sync_or()) break;
    }
    if (tid == 0 && bulk_obs) tc::bulk_wait_all();
    if (bad || abort_flag) {
      abort_flag = 1;
      // cross-play: the tile gave up, so its returns are undefined; NaN (not a stale
      // entry of an earlier call) makes every mean over them NaN
      if (kXp && tid < count) a.xp.returns[env0 + tid] = __int_as_float(0x7FC00000);
    } else if (tid < count) {
      if constexpr (kXp) {
        a.xp.returns[env0 + tid] = Env::ret(st[tid]);
        if (a.xp.steps) a.xp.steps[env0 + tid] = nsteps;
      } else {
        store_state(a.state, N, env_of(tid), st[tid]);
      }
    }
  }

  // ---- drain: every MMA this CTA issued completes (bounded), then free tensor memory ---
  tc::fence_before_sync();
  __syncthreads();
  if (tid == 0 && abort_flag) atomicOr(a.b.status, kStatusTimeout);
  if (warp == 8 && lane == 0) {
    tc::commit(&drain_bar);
    tc::mbar_wait(&drain_bar, 0);
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
  template <bool kXp, bool kSplit, bool kGather>
  static cudaError_t run(const PpoTcArgs& a, int grid, size_t smem, cudaStream_t s) {
    cudaError_t e = cudaFuncSetAttribute(ppo_tc_kernel<Env, kXp, kSplit, kGather>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    ppo_tc_kernel<Env, kXp, kSplit, kGather><<<grid, kTcThreads, smem, s>>>(a);
    return cudaGetLastError();
  }
  // PPO collection with the call's draw (the host keeps IPPO and per-episode teammates of
  // such contexts on CUDA cores)
  static cudaError_t ppo(const PpoTcArgs& a, int grid, size_t smem, cudaStream_t s) {
    const TrajPtrs& u = a.traj1;
    const bool ippo = u.obs || u.actions || u.tm_actions || u.logp || u.values || u.rewards ||
                      u.dones || u.last_value;
    if (!a.tc.sparse || ippo || (a.gather && a.g.resample)) return cudaErrorNotSupported;
    if (a.gather) return a.tc.split ? run<false, true, true>(a, grid, smem, s) : run<false, false, true>(a, grid, smem, s);
    return a.tc.split ? run<false, true, false>(a, grid, smem, s) : run<false, false, false>(a, grid, smem, s);
  }
  static cudaError_t xplay(const PpoTcArgs& a, int grid, size_t smem, cudaStream_t s) {
    if (!a.tc.sparse) return cudaErrorNotSupported;
    return a.tc.split ? run<true, true, false>(a, grid, smem, s) : run<true, false, false>(a, grid, smem, s);
  }
};

}  // namespace aht
