// xplay_tc.cuh -- one step of a cross-play batch whose policies are wide bf16 MLPs
// (hidden width 256 or 512: the Overcooked-style kitchen and Hanabi), with every layer
// contraction on tcgen05 tensor cores and the weights streamed from L2.
//
// The batch holds n_ego x n_tm pairs of P envs each, env e = (i n_tm + j) P + k (ego i,
// teammate j).  One launch is one step s of every env (J_AHT of Sec. 3 estimated per
// pair, XP matrix of App. B).  A tile is up to 128 envs whose acting agent in seat
// `seat` runs the same policy: seat 0 groups the envs of ego i (pairs (i, 0..n_tm-1),
// contiguous), seat 1 those of teammate j (pairs (0..n_ego-1, j)).  For H = 512 a tile
// has two CTAs ("parts", launched as a cluster of two so that they are co-resident): both
// run the transition and the observation; part p computes the N = 256 block p of L1 and
// its epilogue, the parts swap their hidden units' bf16 halves through L2-resident
// exchange slots (a release flag per slot, bounded acquire waits), and part p computes
// block p of L2, its epilogue and that block's share of the output layer -- so each part
// streams half of W1 and half of W2 and runs half of every layer.  The envs
// of a tile change with the seat, so the env state goes through L2 between launches (the
// SoA state, alive flag and actions or output shares are double-buffered by step parity):
//   1. transition: the tile's envs take step s - 1 with the actions the previous launch
//      chose (step 0: reset); with two parts the action is sampled here, from the previous
//      launch's output shares (their sum + b3, masked inverse CDF, Philox stream = seat).
//      Each env has one owning CTA (part 0 of the tile of the seat acting at s, or of the
//      seat-0 tile in simultaneous games) that writes the new state, alive flag, step
//      count and return; the other CTAs compute the same transition for their own use;
//   2. the acting seat's binary observation -> bf16 A operand (exact): its first 512
//      inputs in tensor memory, the rest in shared memory;
//   3. L1 = [o 1] W1^T on tensor cores (one N = 256 block, b1 folded into W1);
//   4. epilogue 1: h1 = tanh(L1), split h1 = hi + lo (two bf16) -> A operands of L2
//      (two parts: each its block's units, then the exchange);
//   5. L2 = hi W2^T + lo W2^T on tensor cores (fp32 accumulate in tensor memory);
//   6. epilogue 2: h2 = tanh(L2 + b2) and this CTA's share of W3 h2 (mma.sync);
//   7. one part: z = W3 h2 + b3 and the masked inverse-CDF sample of the acting seat's
//      action (Philox stream = seat); two parts: the shares go to global memory for the
//      next launch, which adds them and samples.
// Launch max_steps only applies the last transition.
//
// Warp roles (320 threads): warps 0-7 compute (thread r and r + 128 own env row r,
// tensor-memory lane r; the halves split the columns), warp 8 issues the MMAs, warp 9
// streams the 8 KB weight chunks of the tile's policy, in the order the MMAs consume
// them, through a ring of shared-memory stages of several chunks each (one TMA bulk copy
// and one full / empty mbarrier pair per stage).  Every wait is bounded; on expiry the CTA records kStatusTimeout, stops,
// drains its MMAs and copies, frees tensor memory and exits.
//
// Tensor memory (512 columns), R0 = [0, 256), R1 = [256, 512); the observation's first
// 512 inputs sit in R1 until L1 is done:
//   H = 256: L1 -> R0; epilogue 1 rewrites each 32-column block of R0 in place as
//            16 columns hi | 16 columns lo; L2 -> R1.
//   H = 512: L1 block `part` -> R0; epilogue 1 writes hi to shared memory (a [128][512]
//            canonical A operand over the dead observation tile) and, after the
//            exchange, lo of all 512 units packed into R0; L2 block `part` -> R1.
#pragma once
#include "kernels.h"
#include "mlp_simt.cuh"
#include "rollout_impl.cuh"
#include "tc_common.cuh"

namespace aht {

constexpr int kXpCompute = 256;
constexpr int kXpThreads = 320;
constexpr int kXpComputeBar = 1;
constexpr int kXpMaxStages = 3;
constexpr int kXpMaxChunksPerStage = 12;  // a bulk copy's rate grows with its size (to ~100 KB)
constexpr uint32_t kXpSmemBudget = 231424;  // opt-in maximum minus a margin for static data

struct XpTcSmem {
  uint32_t a_bytes;    // env states / observation tile / hi operand, W3 b2 b3, partials
  uint32_t w3_off;     // W3, b2, b3 (bulk-copied once L1 is done), within the A region
  uint32_t w3_bytes;
  uint32_t stage_off;  // weight stages
  uint32_t bits_off;   // per-row observation bits: the tail of the stage area, dead once the
                       // observation is expanded (stages overlapping it are filled after that)
  uint32_t total;
  int nst;             // stages
  int spc;             // 8 KB chunks per stage (one bulk copy, one full / empty barrier pair)
  int bit_words;       // 32-bit words per observation bit row
  int k_tm;            // the first k_tm observation inputs form L1's A operand in tensor
                       // memory (columns [256, 256 + k_tm / 2), free until L2); the rest
                       // (KP - k_tm) sit in shared memory
};

__host__ __device__ inline XpTcSmem xp_tc_layout(const WideDims& w) {
  XpTcSmem L;
  // L1: observation tile, only its part beyond the tensor-memory columns (L1's accumulator
  // takes 256 columns: all units for H = 256, this part's block for H = 512).  L2 and
  // after: hi (H = 512) or the output partials, then W3.
  L.k_tm = w.KP < 512 ? w.KP : 512;
  const uint32_t obs = 128u * (uint32_t)(w.KP - L.k_tm) * 2u;
  const uint32_t hi = w.H == 512 ? 128u * 512u * 2u : 0u;
  const uint32_t zp = 2u * 128u * (uint32_t)w.NAP * 4u;
  L.w3_off = (uint32_t)align_up(hi > zp ? hi : zp, 1024);
  L.w3_bytes = w.pol_bytes - w.oW3;
  const uint32_t a = L.w3_off + L.w3_bytes > obs ? L.w3_off + L.w3_bytes : obs;
  L.a_bytes = (uint32_t)align_up(a, 1024);
  L.bit_words = (w.KP + 31) / 32;
  const uint32_t bits = (uint32_t)align_up(128 * L.bit_words * 4, 1024);
  // Two stages as large as fit: on GB300 a bulk copy takes about the same 500-2000 cycles
  // to land for 8 KB as for 32 KB, and copies in flight barely overlap (measured, also
  // with several issuing warps), so the bytes per copy set the stream's rate.
  // The observation bits share the last stage's space when that buys larger stages (they
  // are dead once the observation is expanded), else they sit after the stages.
  auto config = [&](int slots, int& spc, int& nst) {
    spc = slots / 2 > kXpMaxChunksPerStage ? kXpMaxChunksPerStage : slots / 2;
    nst = slots / spc > kXpMaxStages ? kXpMaxStages : slots / spc;
  };
  int spc_s, nst_s, spc_a, nst_a;
  config((int)((kXpSmemBudget - L.a_bytes - bits) / kWideChunk), spc_s, nst_s);
  config((int)((kXpSmemBudget - L.a_bytes) / kWideChunk), spc_a, nst_a);
  const bool alias = spc_a * nst_a > spc_s * nst_s;
  L.spc = alias ? spc_a : spc_s;
  L.nst = alias ? nst_a : nst_s;
  L.stage_off = L.a_bytes;
  const uint32_t stages_end = L.stage_off + (uint32_t)(L.nst * L.spc) * kWideChunk;
  L.bits_off = alias ? stages_end - bits : stages_end;
  L.total = alias ? stages_end : stages_end + bits;
  return L;
}

// Two binary features (bits 0, 1 of x) as a bf16 pair: 0 or 1.0 (0x3F80) each.  Bit 0
// times 0x8001 stays at bit 0 and bit 1 lands on bit 16 (the mask drops the cross terms),
// so one multiply by 0x3F80 writes both halves.
__device__ __forceinline__ uint32_t bits_to_bf16x2(uint32_t x) {
  return (((x & 3u) * 0x8001u) & 0x00010001u) * 0x3F80u;
}

// The parts of a tile publish their exchange slot with a release store of the flag after
// a barrier of the writing threads (one thread, after a gpu-scope fence), and the reader
// polls it with acquire loads and then releases its threads with a barrier.
__device__ __forceinline__ void xch_publish(uint32_t* flag, uint32_t v) {
  asm volatile("fence.acq_rel.gpu;\nst.relaxed.gpu.global.u32 [%0], %1;" ::"l"(flag), "r"(v) : "memory");
}
// Until *flag is `ok` (true) or ok + 1 (the writer gave up: false); false as well after 2 s.
__device__ __forceinline__ bool xch_wait(const uint32_t* flag, uint32_t ok) {
  const uint64_t t0 = tc::globaltimer_ns();
  for (uint32_t i = 0; i < (1u << 30); ++i) {
    uint32_t v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(flag) : "memory");
    if (v == ok) return true;
    if (v == ok + 1u) return false;
    if ((i & 63u) == 63u && tc::globaltimer_ns() - t0 > 2000000000ull) return false;
  }
  return false;
}

template <class Env>
__global__ void __launch_bounds__(kXpThreads, 1) xp_tc_kernel(const XpTcArgs a) {
  using State = typename Env::State;
  constexpr int NA = Env::kNumActions;
  constexpr int NAP = (NA + 3) / 4 * 4;
  constexpr bool kTurn = Env::kTurnBased;
  extern __shared__ __align__(16) uint8_t smem[];  // the no-swizzle operands need 16 B
  __shared__ __align__(8) uint64_t full_bar[kXpMaxStages], empty_bar[kXpMaxStages];
  __shared__ __align__(8) uint64_t obs_bar, acc_bar[3], epi1_bar, epi2_bar, w3_bar, drain_bar;
  __shared__ __align__(8) uint64_t never_bar;  // test hook: nothing arrives on it
  __shared__ uint32_t tmem_slot;
  __shared__ volatile int abort_flag;
  bool w3_issued = false;  // (MMA lane) the W3 copy is in flight or done
  int next_chunk = 0;      // (producer lane) stages issued

  const WideDims& w = a.w;
  const XpTcSmem L = xp_tc_layout(w);
  const int NST = L.nst;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, row = tid & 127;
  const int half = (warp >> 2) & 1;

  // ---- the tile: seat, acting policy, rows ------------------------------------------
  const int G0 = a.n_tm * a.P, G1 = a.n_ego * a.P;
  const int T0 = (G0 + 127) / 128, T1 = (G1 + 127) / 128;
  // a.parts CTAs per tile: part p computes layer 2's N = 256 block p (H = 512, two parts)
  int seat, t = (int)blockIdx.x / a.parts;
  const int part = (int)blockIdx.x - t * a.parts;
  if (kTurn) {
    seat = a.s & 1;
  } else {
    seat = t < a.n_ego * T0 ? 0 : 1;
    if (seat) t -= a.n_ego * T0;
  }
  const int Tn = seat ? T1 : T0, G = seat ? G1 : G0;
  const int group = t / Tn, q0 = (t - group * Tn) * 128;
  const int count = min(128, G - q0);
  const int pol = seat ? a.tm_ids[group] : a.ego_ids[group];
  const bool owner = (kTurn || seat == 0) && part == 0;  // writes the envs' state and records
  auto env_of = [&](int r) -> int64_t {
    const int q = q0 + r;
    if (seat == 0) return (int64_t)group * G0 + q;
    const int i = q / a.P, k = q - i * a.P;
    return ((int64_t)i * a.n_tm + group) * a.P + k;
  };

  uint8_t* const sA = smem;
  uint8_t* const sStage = smem + L.stage_off;
  uint32_t* const sBits = reinterpret_cast<uint32_t*>(smem + L.bits_off);
  const uint8_t* const pblk = a.tcw + (int64_t)pol * w.pol_bytes;
  const uint32_t gt = a.step0 + (uint32_t)a.s;

  // ---- 0. overlap with the previous step's launch (programmatic dependent launch) ------
  // The next step's CTAs may start now; everything up to griddepcontrol.wait touches
  // nothing the previous step writes (barriers, tensor memory).
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  if (tid == 0) {
    for (int i = 0; i < NST; ++i) {
      tc::mbar_init(&full_bar[i], 1);
      tc::mbar_init(&empty_bar[i], 1);
    }
    tc::mbar_init(&obs_bar, kXpCompute);
    for (int i = 0; i < 3; ++i) tc::mbar_init(&acc_bar[i], 1);
    tc::mbar_init(&epi1_bar, kXpCompute);
    tc::mbar_init(&epi2_bar, kXpCompute);
    tc::mbar_init(&w3_bar, 1);
    tc::mbar_init(&drain_bar, 1);
    tc::mbar_init(&never_bar, 1);
    tc::mbar_init_fence();
    abort_flag = 0;
  }
  if (warp == 0) tc::tmem_alloc(&tmem_slot, 512);
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  // the chunks this CTA streams: W1's, then W2's -- with two parts only block `part` of
  // each (N = 256 rows of W1 and of W2); chunk c of the stream is chunk src(c) of the
  // policy block
  const int n_l1_own = w.n_l1 / a.parts, n_l2_own = w.n_l2 / a.parts;
  const int n_chunks = n_l1_own + n_l2_own;
  const int SPC = L.spc, n_stages = (n_chunks + SPC - 1) / SPC;
  const uint32_t stage_bytes = (uint32_t)SPC * kWideChunk;
  auto src_chunk = [&](int c) {  // W1 block `part`, then W2 block `part`
    return c < n_l1_own ? part * n_l1_own + c : w.n_l1 + part * n_l2_own + (c - n_l1_own);
  };
  // stage k -> one bulk copy, or two where it straddles the W1 / W2 boundary
  auto copy_stage = [&](int k, uint8_t* dst, uint64_t* bar, uint64_t policy) {
    const int c0 = k * SPC, c1 = min(c0 + SPC, n_chunks);
    tc::mbar_expect_tx(bar, (uint32_t)(c1 - c0) * kWideChunk);
    const int cut = c0 < n_l1_own && c1 > n_l1_own ? n_l1_own : c1;  // end of the first piece
    tc::bulk_g2s_hint(dst, pblk + (int64_t)src_chunk(c0) * kWideChunk, (uint32_t)(cut - c0) * kWideChunk, bar,
                      policy);
    if (cut < c1)
      tc::bulk_g2s_hint(dst + (size_t)(cut - c0) * kWideChunk, pblk + (int64_t)src_chunk(cut) * kWideChunk,
                        (uint32_t)(c1 - cut) * kWideChunk, bar, policy);
  };
  // producer state (warp 9, lane 0): next stage, its ring slot, uses of that slot so far
  int pk = 0, pslot = 0;
  uint32_t puse = 0;
  // stages whose slot ends at or below the observation bits may be filled at once
  const int free_slots = (int)((L.bits_off - L.stage_off) / stage_bytes);
  if (warp == 9 && lane == 0) {  // the first stages: the population is read-only
    const uint64_t keep = tc::l2_evict_last();
    for (; pk < n_stages && pk < NST && pk < free_slots; ++pk, ++pslot)
      copy_stage(pk, sStage + pslot * stage_bytes, &full_bar[pslot], keep);
    if (pslot == NST) {
      pslot = 0;
      puse = 1;
    }
  }
  // the previous step's state, alive flags and actions are complete and visible
  asm volatile("griddepcontrol.wait;" ::: "memory");

  // ---- 1. transition of step s - 1, and this step's observation bits -----------------
  bool alive = false;
  int64_t e = -1;
  float u_act = 0.0f;                           // one part: this step's sampling happens here
  uint32_t legal = 0xFFFFFFFFu >> (32 - NA);
  // Two parts: the action seat q of env e chose at step s - 1 comes from the outputs of the
  // previous launch -- the two parts' shares plus b3 of seat q's policy -- sampled as in
  // every other kernel (masked inverse CDF, Philox stream q at step s - 1).  The shares
  // and b3 are loaded (16-byte vectors) before the state, so their latency overlaps it.
  constexpr int kActing = kTurn ? 1 : 2;  // seats that act in a step
  auto gather_z = [&](int q, int64_t env, float (&z)[NAP]) {  // false if a part gave up (NaN)
    const float4* zp = reinterpret_cast<const float4*>(a.zp_in + ((env * 2 + q) * 2) * NAP);
    const uint32_t pair = (uint32_t)env / (uint32_t)a.P;  // 32-bit: n_total < 2^31
    const int i = (int)(pair / (uint32_t)a.n_tm), j = (int)(pair - (uint32_t)i * (uint32_t)a.n_tm);
    const int pq = q == 0 ? a.ego_ids[i] : a.tm_ids[j];
    const float4* b3 = reinterpret_cast<const float4*>(a.tcw + (int64_t)pq * w.pol_bytes + w.ob3);
#pragma unroll
    for (int v = 0; v < NAP / 4; ++v) {
      const float4 p0 = zp[v], p1 = zp[NAP / 4 + v], bb = b3[v];
      z[4 * v] = (p0.x + p1.x) + bb.x;
      z[4 * v + 1] = (p0.y + p1.y) + bb.y;
      z[4 * v + 2] = (p0.z + p1.z) + bb.z;
      z[4 * v + 3] = (p0.w + p1.w) + bb.w;
    }
  };
  auto pick = [&](int q, const State& st, int64_t env, const float (&z)[NAP]) -> int {
    bool finite = true;
#pragma unroll
    for (int o = 0; o < NAP; ++o) finite = finite && z[o] == z[o];
    if (!finite) return -1;
    if (owner && a.dbg_logits) {  // test hook: the outputs of step s - 1
      float* p = a.dbg_logits + (((int64_t)(a.s - 1) * a.n_total + env) * 2 + q) * kDbgStride;
#pragma unroll
      for (int o = 0; o < NAP; ++o) p[o] = z[o];
    }
    const uint32_t lg = kTurn ? Env::legal(st) : 0xFFFFFFFFu >> (32 - NA);
    const float u = u01(draw0(a.b.key, (uint32_t)env, gt - 1u, kStreamAct0 + q));
    float lp;
    return sample_k<NA>(z, lg, u, lp);
  };
  if (tid < 128) {
    uint32_t* bits = sBits + row * L.bit_words;
    if (row < count) {
      e = env_of(row);
      // the state lives in shared memory (the A region is free until the observation is
      // expanded): per-thread local copies would spill past the small L1 left beside
      // this kernel's shared memory
      State& s = reinterpret_cast<State*>(sA)[row];
      int nst = 0;
      const int actor = kTurn ? ((a.s - 1) & 1) : -1;  // the seat that acted at s - 1
      float zq[kActing][NAP];
      const bool two = a.parts == 2 && a.s > 0;
      if (two) {
#pragma unroll
        for (int k = 0; k < kActing; ++k) gather_z(kTurn ? actor : k, e, zq[k]);
      }
      if (a.s == 0) {
        Env::reset(a.b.env, a.b.key, (uint32_t)e, a.step0, s);
        alive = true;
      } else {
        load_state(a.st_in, a.n_total, e, s);
        alive = a.alive_in[e] != 0;
        if (owner) nst = a.nsteps[e];
        if (alive) {
          int a0 = 0, a1 = 0;
          if (two) {
            if (kTurn) {
              const int act = pick(actor, s, e, zq[0]);
              (actor == 0 ? a0 : a1) = act;
              if (act < 0) a0 = -1;
            } else {
              a0 = pick(0, s, e, zq[0]);
              a1 = pick(1, s, e, zq[kActing - 1]);
            }
          } else {
            if (actor < 0 || actor == 0) a0 = a.act_in[2 * e];
            if (actor < 0 || actor == 1) a1 = a.act_in[2 * e + 1];
          }
          if (a0 < 0 || a1 < 0) {
            alive = false;  // a part of the previous launch gave up: the env stops
          } else {
            if (owner && a.actions) {
              uint8_t* rec = a.actions + ((int64_t)(a.s - 1) * a.n_total + e) * 2;
              rec[0] = (actor < 0 || actor == 0) ? (uint8_t)a0 : 255;
              rec[1] = (actor < 0 || actor == 1) ? (uint8_t)a1 : 255;
            }
            float r0, r1, team;
            const int done = Env::step(a.b.env, s, a0, a1, r0, r1, team);
            if (done < 0) {
              if (owner) atomicOr(a.b.status, kStatusIllegalAction);
              alive = false;
            } else {
              nst += 1;
              if (done) alive = false;
            }
          }
        }
      }
      if (owner) {
        store_state(a.st_out, a.n_total, e, s);
        a.alive_out[e] = (uint8_t)alive;
        a.nsteps[e] = nst;
        a.returns[e] = Env::ret(s);
        if (a.steps) a.steps[e] = nst;
      }
      if (alive && a.s < a.max_steps) {
        ObsBits wr{bits, L.bit_words};
        Env::obs_into(a.b.env, s, seat, wr);
        wr.set(a.b.env.obs_dim, 1);  // the constant input that carries b1
        if (kTurn) {
          legal = Env::legal(s);
          if (Env::actor(s) != seat) atomicOr(a.b.status, kStatusActorMismatch);
        }
        if (a.parts == 1) u_act = u01(draw0(a.b.key, (uint32_t)e, gt, kStreamAct0 + seat));
      } else {
        for (int i = 0; i < L.bit_words; ++i) bits[i] = 0u;
      }
    } else {
      for (int i = 0; i < L.bit_words; ++i) bits[i] = 0u;
    }
  }
  tc::fence_before_sync();
  const bool proceed = __syncthreads_or(alive) && a.s < a.max_steps;
  tc::fence_after_sync();
  const uint32_t tmem = tmem_slot;
  if (!proceed) {  // nothing left to act this step: the prefetched stages land, then exit
    if (warp == 9 && lane == 0)
      for (int d = 0; d < pk; ++d) tc::mbar_wait(&full_bar[d], 0u);
    if (warp == 0) tc::tmem_dealloc(tmem, 512);
    return;
  }
  if (warp == 9) {
    // ============================ weight producer ===================================
    if (lane == 0) {
      int k = pk, slot = pslot;  // continues after the prefetched stages
      uint32_t use = puse;       // times the slot was filled before
      bool ok = true, obs_seen = false;
      const uint64_t keep = tc::l2_evict_last();  // every step re-reads the population
      for (; k < n_stages; ++k) {
        if (use == 0 && slot >= free_slots && !obs_seen) {  // the bits are read by then
          ok = false;
          for (int tries = 0; tries < 1000 && !ok && !abort_flag; ++tries)
            ok = tc::mbar_wait(&obs_bar, 0u, 2000000ull);
          if (!ok) break;
          obs_seen = true;
        }
        if (use > 0) {
          ok = false;
          for (int tries = 0; tries < 1000 && !ok && !abort_flag; ++tries)
            ok = tc::mbar_wait(&empty_bar[slot], (use - 1) & 1u, 2000000ull);
          if (!ok) break;
        }
        copy_stage(k, sStage + slot * stage_bytes, &full_bar[slot], keep);
        if (++slot == NST) {
          slot = 0;
          ++use;
        }
      }
      if (!ok) abort_flag = 1;
      next_chunk = k;  // stages issued
    }
  } else if (warp == 8) {
    // ================================ MMA issue =====================================
    if (lane == 0) {
      const uint32_t idesc = tc::idesc_bf16(128, 256);
      auto wait_for = [&](uint64_t* bar, uint32_t parity) {
        bool ok = false;
        for (int tries = 0; tries < 1000 && !ok && !abort_flag; ++tries)
          ok = tc::mbar_wait(bar, parity, 2000000ull);
        if (ok) tc::fence_after_sync();
        return ok;
      };
      // ring cursor of the next chunk: its stage's slot, its position in the stage, the
      // slot's full-barrier parity; advanced by increments (a runtime division per chunk
      // costs this single thread hundreds of cycles)
      int c = 0, sub = 0, slot = 0;
      uint32_t fpar = 0;
      const uint32_t stage0 = tc::smem_u32(sStage);
      auto chunk = [&](uint64_t& desc) {  // waits for weight chunk c, returns its descriptor
        if (sub == 0 && !wait_for(&full_bar[slot], fpar)) return false;
        desc = tc::smem_desc(stage0 + (uint32_t)slot * stage_bytes + (uint32_t)sub * kWideChunk, 128u, 256u);
        return true;
      };
      auto release = [&]() {  // the stage is free once the MMAs reading its last chunk finish
        if (++sub == SPC || c == n_chunks - 1) {
          tc::commit(&empty_bar[slot]);
          sub = 0;
          if (++slot == NST) {
            slot = 0;
            fpar ^= 1u;
          }
        }
        ++c;
      };
      bool ok = wait_for(&obs_bar, 0);
      // L1: one N = 256 block (all units for H = 256, block `part` for H = 512) into
      // columns [0, 256); the observation operand has inputs [0, k_tm) in tensor memory,
      // the rest in shared memory as a canonical [128][KP - k_tm] matrix
      const int ks_tm = L.k_tm / 16;
      const uint32_t aobs = tc::smem_u32(sA), sbo_obs = (uint32_t)((w.KP - L.k_tm) / 8) * 128u;
      for (int ks = 0; ok && ks < w.KP / 16; ++ks) {
        uint64_t bd;
        if (!(ok = chunk(bd))) break;
        if (ks < ks_tm)
          tc::mma_ts(tmem, tmem + 256u + 8u * ks, bd, idesc, ks > 0);
        else
          tc::mma_ss(tmem, tc::smem_desc(aobs + 256u * (ks - ks_tm), 128u, sbo_obs), bd, idesc, ks > 0);
        release();
      }
      if (ok) tc::commit(&acc_bar[0]);
      // once L1 has read the observation tile, W3 b2 b3 go to the A region's tail
      if (ok) ok = wait_for(&acc_bar[0], 0);
      if (ok) {
        tc::mbar_expect_tx(&w3_bar, L.w3_bytes);
        tc::bulk_g2s(sA + L.w3_off, pblk + w.oW3, L.w3_bytes, &w3_bar);
        w3_issued = true;
      }
      if (ok) ok = wait_for(&epi1_bar, 0);
      if (ok && w.H == 256) {
        for (int ks = 0; ok && ks < 16; ++ks) {
          uint64_t bd;
          if (!(ok = chunk(bd))) break;
          const uint32_t hi = tmem + 32u * (ks >> 1) + 8u * (ks & 1);
          tc::mma_ts(tmem + 256u, hi, bd, idesc, ks > 0);
          tc::mma_ts(tmem + 256u, hi + 16u, bd, idesc, 1u);
          release();
        }
        if (ok) tc::commit(&acc_bar[1]);
      } else if (ok) {
        const uint32_t ahi = tc::smem_u32(sA);
        // this CTA's blocks of L2: both, or its part's (then into acc_bar[1])
        const int nh0 = a.parts == 2 ? part : 0, nh1 = a.parts == 2 ? part + 1 : 2;
        for (int nh = nh0; ok && nh < nh1; ++nh) {
          if (nh > nh0 && !(ok = wait_for(&epi2_bar, 0))) break;
          for (int ks = 0; ok && ks < 32; ++ks) {
            uint64_t bd;
            if (!(ok = chunk(bd))) break;
            tc::mma_ss(tmem + 256u, tc::smem_desc(ahi + 256u * ks, 128u, 64u * 128u), bd, idesc, ks > 0);
            tc::mma_ts(tmem + 256u, tmem + 8u * ks, bd, idesc, 1u);
            release();
          }
          if (ok) tc::commit(&acc_bar[1 + nh - nh0]);
        }
      }
      if (!ok) abort_flag = 1;
    }
  } else {
    // ============================== compute warps ===================================
    bool bad = false;
    const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;
    const uint32_t R0 = tmem + lane_base;
    auto wait_acc = [&](uint64_t* bar) {
      if (!bad && !tc::mbar_wait(bar, 0)) bad = true;
      bad = __any_sync(0xFFFFFFFFu, bad);
      tc::fence_after_sync();
    };
    auto sync_or = [&]() { return tc::bar_or(kXpComputeBar, kXpCompute, bad || abort_flag); };

    // 2. observation bits -> bf16 A operand.  H = 512: all in shared memory (canonical
    //    K-major [128][KP]).  H = 256: 8-feature blocks [0, k_tm / 8) into tensor memory
    //    (this warp's rows, 4 columns per block, two blocks per store), the rest into
    //    shared memory ([128][KP - k_tm]).  Each half of the threads expands an even-sized
    //    half of the row's blocks.
    {
      const uint32_t* bits = sBits + row * L.bit_words;
      const int nkb = w.KP / 8, split = (nkb / 2) & ~1, kb_tm = L.k_tm / 8;
      const int kb0 = half ? split : 0, kb1 = half ? nkb : split;
      auto block = [&](uint32_t word, int kb, uint32_t (&v)[4]) {  // block kb's bf16 pairs
        const uint32_t byte = (word >> (8 * (kb & 3))) & 0xFFu;  // word = bits[kb / 4]
        v[0] = bits_to_bf16x2(byte);
        v[1] = bits_to_bf16x2(byte >> 2);
        v[2] = bits_to_bf16x2(byte >> 4);
        v[3] = bits_to_bf16x2(byte >> 6);
      };
      int kb = kb0;
      if (kb_tm > 0) {
        // KP and k_tm are multiples of 16 and `split` is even, so each half's blocks in
        // tensor memory come in pairs (kb even: column 256 + 4 kb is a multiple of 8)
        const int t1 = kb1 < kb_tm ? kb1 : kb_tm;
        for (; kb < t1; kb += 2) {
          const uint32_t word = bits[kb >> 2];  // kb even: kb + 1 is in the same word
          uint32_t v[8], u[4];
          block(word, kb, u);
          v[0] = u[0], v[1] = u[1], v[2] = u[2], v[3] = u[3];
          block(word, kb + 1, u);
          v[4] = u[0], v[5] = u[1], v[6] = u[2], v[7] = u[3];
          tc::st_x8(tmem + lane_base + 256u + 4u * (uint32_t)kb, v);
        }
        tc::wait_st();
        if (kb < kb_tm) kb = kb_tm;
      }
      // the shared-memory part: 16-byte core-matrix rows of consecutive blocks 128 bytes apart
      uint8_t* dst = sA + tc::canon_offset(row, 8 * (kb - kb_tm), w.KP - L.k_tm);
      uint32_t word = kb < kb1 ? bits[kb >> 2] : 0u;
      for (; kb < kb1; ++kb, dst += 128) {
        if ((kb & 3) == 0) word = bits[kb >> 2];
        uint4 v;
        v.x = bits_to_bf16x2(word >> (8 * (kb & 3)));
        v.y = bits_to_bf16x2(word >> (8 * (kb & 3) + 2));
        v.z = bits_to_bf16x2(word >> (8 * (kb & 3) + 4));
        v.w = bits_to_bf16x2(word >> (8 * (kb & 3) + 6));
        *reinterpret_cast<uint4*>(dst) = v;
      }
      tc::fence_proxy_async();
      if (kb_tm > 0) tc::fence_before_sync();
      tc::mbar_arrive(&obs_bar);
    }

    // 4. epilogue 1
    if (a.s == a.dbg_expire_step) {  // test hook: an accumulator wait that never completes
      if (!bad && !tc::mbar_wait(&never_bar, 0, a.dbg_expire_ns)) bad = true;
      bad = __any_sync(0xFFFFFFFFu, bad);
    }
    wait_acc(&acc_bar[0]);
    if (!bad && w.H == 256) {
      for (int c0 = 128 * half; c0 < 128 * half + 128; c0 += 32) {
        uint32_t v[32], hi[16], lo[16];
        tc::ld_x32(R0 + c0, v);
        tc::wait_ld();
#pragma unroll
        for (int j = 0; j < 16; ++j)
          tc::split_bf16x2_p(tc::tanh2(tc::f2_pack(__uint_as_float(v[2 * j]), __uint_as_float(v[2 * j + 1]))),
                             hi[j], lo[j]);
        tc::st_x16(R0 + c0, hi);
        tc::st_x16(R0 + c0 + 16, lo);
      }
      tc::wait_st();
    } else if (w.H == 512) {
      // This part's block of L1, units [256 part, 256 part + 256) in R0 [0, 256); half h
      // takes [128 h, 128 h + 128) of it.  hi -> shared memory (the canonical [128][512]
      // A operand of L2) and this CTA's exchange slot; lo -> the slot and registers.  Then
      // the two parts of the tile swap halves through L2-resident memory: each takes the
      // other's hi into shared memory, and every unit's lo goes to R0 packed (unit u at
      // column u / 2) once all of R0 has been read.
      uint32_t lo_keep[64];
      uint4* const mine = reinterpret_cast<uint4*>(a.xch + (size_t)blockIdx.x * kXchSlot);
      for (int cb = 0; cb < 4; ++cb) {
        if (bad) break;
        uint32_t v[32], hi[16];
        tc::ld_x32(R0 + 128u * half + 32u * cb, v);
        tc::wait_ld();
#pragma unroll
        for (int j = 0; j < 16; ++j)
          tc::split_bf16x2_p(tc::tanh2(tc::f2_pack(__uint_as_float(v[2 * j]), __uint_as_float(v[2 * j + 1]))),
                             hi[j], lo_keep[16 * cb + j]);
        const int ub = 128 * half + 32 * cb;  // unit within the block
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const uint4 h4 = make_uint4(hi[4 * q], hi[4 * q + 1], hi[4 * q + 2], hi[4 * q + 3]);
          *reinterpret_cast<uint4*>(sA + tc::canon_offset(row, 256 * part + ub + 8 * q, 512)) = h4;
          const int ch = ub / 8 + q;  // 8-unit chunk of the block
          __stcg(mine + ch * 128 + row, h4);
          __stcg(mine + (32 + ch) * 128 + row,
                 make_uint4(lo_keep[16 * cb + 4 * q], lo_keep[16 * cb + 4 * q + 1], lo_keep[16 * cb + 4 * q + 2],
                            lo_keep[16 * cb + 4 * q + 3]));
        }
      }
      // publish this part's slot (2 stamp, or 2 stamp + 1 when it gave up), then take the
      // partner's (bounded wait; a partner that gave up makes this part give up too)
      tc::fence_before_sync();
      bad = sync_or();  // also: every thread has read its columns of R0
      tc::fence_after_sync();
      const uint32_t partner = blockIdx.x ^ 1u;
      if (tid == 0) {
        xch_publish(a.xflag + blockIdx.x, 2u * a.xstamp + (bad ? 1u : 0u));
        if (!bad && !xch_wait(a.xflag + partner, 2u * a.xstamp)) bad = true;
      }
      bad = sync_or();
      if (!bad) {
        const uint4* const theirs = reinterpret_cast<const uint4*>(a.xch + (size_t)partner * kXchSlot);
        const int op = 1 - part;
        // the partner's hi for units [256 op + 128 h, + 128) of this row
#pragma unroll 4
        for (int q = 0; q < 16; ++q)
          *reinterpret_cast<uint4*>(sA + tc::canon_offset(row, 256 * op + 128 * half + 8 * q, 512)) =
              __ldcg(theirs + (16 * half + q) * 128 + row);
        // lo: this thread's own units -> columns [128 part + 64 h, + 64), the partner's
        // units [256 op + 128 h, + 128) -> columns [128 op + 64 h, + 64)
        tc::st_x32(R0 + 128u * part + 64u * half, *reinterpret_cast<const uint32_t(*)[32]>(lo_keep));
        tc::st_x32(R0 + 128u * part + 64u * half + 32u, *reinterpret_cast<const uint32_t(*)[32]>(lo_keep + 32));
#pragma unroll
        for (int g2 = 0; g2 < 2; ++g2) {
          uint32_t v[32];
#pragma unroll
          for (int q = 0; q < 8; ++q) {
            const uint4 l4 = __ldcg(theirs + (32 + 16 * half + 8 * g2 + q) * 128 + row);
            v[4 * q] = l4.x, v[4 * q + 1] = l4.y, v[4 * q + 2] = l4.z, v[4 * q + 3] = l4.w;
          }
          tc::st_x32(R0 + 128u * op + 64u * half + 32u * g2, v);
        }
        tc::wait_st();
      }
    }
    tc::fence_proxy_async();  // hi written by ordinary stores, read by the tensor cores
    tc::fence_before_sync();
    tc::mbar_arrive(&epi1_bar);

    // 6. epilogue 2: this half's columns of each N = 256 block of L2
    const float* W3 = reinterpret_cast<const float*>(sA + L.w3_off);
    const float* b2 = reinterpret_cast<const float*>(sA + L.w3_off + (w.ob2 - w.oW3));
    const float* b3 = reinterpret_cast<const float*>(sA + L.w3_off + (w.ob3 - w.oW3));
    if (!bad && !tc::mbar_wait(&w3_bar, 0)) bad = true;
    bad = __any_sync(0xFFFFFFFFu, bad);
    // The output layer on the tensor cores from registers (mma.sync m16n8k16): each warp
    // takes its 32 rows as two groups of 16 and its half's 128 units of each N = 256
    // block as chunks of 16.  Two 16x256b loads of the accumulator give the thread the
    // values of the A fragment (rows g, g + 8; units 2c, 2c + 1 and 2c + 8, 2c + 9 of the
    // chunk, g = lane / 4, c = lane % 4); h2 = tanh(acc + b2) is split h2 = hi + lo (two
    // bf16) and z accumulates hi W3^T + lo W3^T in fp32, n-tiles of 8 outputs.
    constexpr int NT = (NAP + 7) / 8;
    const uint32_t* W3f = reinterpret_cast<const uint32_t*>(W3);
    const int g = lane >> 2, c4 = lane & 3;
    float zacc[2][NT][4];
#pragma unroll
    for (int rg = 0; rg < 2; ++rg)
#pragma unroll
      for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int i = 0; i < 4; ++i) zacc[rg][nt][i] = 0.0f;
    // the N = 256 blocks of L2 this CTA computes: all, or its part's
    const int nb0 = a.parts == 2 ? part : 0, nb1 = a.parts == 2 ? part + 1 : w.H / 256;
    const uint32_t R1q = tmem + 256u + ((uint32_t)((warp & 3) * 32) << 16);  // this warp's rows
    for (int nh = nb0; nh < nb1; ++nh) {
      wait_acc(&acc_bar[1 + nh - nb0]);
      if (bad) break;
#pragma unroll 1
      for (int kc = 0; kc < 8; ++kc) {
        const int c0 = 128 * half + 16 * kc;             // column of the N = 256 block
        const int u0 = 256 * nh + c0;                    // hidden unit
        const int j = u0 / 16;                           // W3 chunk
        const uint64_t bA = *reinterpret_cast<const uint64_t*>(b2 + u0 + 2 * c4);
        const uint64_t bB = *reinterpret_cast<const uint64_t*>(b2 + u0 + 8 + 2 * c4);
#pragma unroll
        for (int rg = 0; rg < 2; ++rg) {
          uint32_t t0[4], t1[4];
          tc::ld_16x256b(R1q + ((uint32_t)(16 * rg) << 16) + (uint32_t)c0, t0);
          tc::ld_16x256b(R1q + ((uint32_t)(16 * rg) << 16) + (uint32_t)(c0 + 8), t1);
          tc::wait_ld();
          uint32_t ahi[4], alo[4];
          tc::split_bf16x2_p(tc::tanh2(tc::f2_add(tc::f2_pack(__uint_as_float(t0[0]), __uint_as_float(t0[1])), bA)),
                             ahi[0], alo[0]);
          tc::split_bf16x2_p(tc::tanh2(tc::f2_add(tc::f2_pack(__uint_as_float(t0[2]), __uint_as_float(t0[3])), bA)),
                             ahi[1], alo[1]);
          tc::split_bf16x2_p(tc::tanh2(tc::f2_add(tc::f2_pack(__uint_as_float(t1[0]), __uint_as_float(t1[1])), bB)),
                             ahi[2], alo[2]);
          tc::split_bf16x2_p(tc::tanh2(tc::f2_add(tc::f2_pack(__uint_as_float(t1[2]), __uint_as_float(t1[3])), bB)),
                             ahi[3], alo[3]);
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) {
            const uint2 bw = *reinterpret_cast<const uint2*>(W3f + ((j * NT + nt) * 32 + lane) * 2);
            tc::mma_m16n8k16_bf16(zacc[rg][nt], ahi, bw.x, bw.y);
            tc::mma_m16n8k16_bf16(zacc[rg][nt], alo, bw.x, bw.y);
          }
        }
      }
      if (nh + 1 < nb1) {
        tc::fence_before_sync();
        tc::mbar_arrive(&epi2_bar);  // R1 may take the second half
      }
    }
    // partial sums of the two halves -> shared memory (the A region is dead now)
    float* zpart = reinterpret_cast<float*>(sA);
    if (!bad) {
#pragma unroll
      for (int rg = 0; rg < 2; ++rg) {
        const int r0 = 32 * (warp & 3) + 16 * rg + g;
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const int o = 8 * nt + 2 * c4 + (i & 1), r = r0 + 8 * (i >> 1);
            if (o < NAP) zpart[(half * 128 + r) * NAP + o] = zacc[rg][nt][i];
          }
      }
    }
    bad = sync_or();

    // 7. one part: sample the acting seat's action (half 0 threads, live rows).  Two parts:
    //    this CTA's share of the outputs (the sum over its units of W3 h2) goes to global
    //    memory, and the next launch adds the shares and b3 and samples.
    if (a.parts == 1) {
      if (!bad && tid < 128 && alive) {
        float z[NAP];
#pragma unroll
        for (int o = 0; o < NAP; ++o)
          z[o] = (zpart[row * NAP + o] + zpart[(128 + row) * NAP + o]) + b3[o];
        if (a.dbg_logits) {  // test hook: this row's outputs of step s
          float* p = a.dbg_logits + (((int64_t)a.s * a.n_total + e) * 2 + seat) * kDbgStride;
#pragma unroll
          for (int o = 0; o < NAP; ++o) p[o] = z[o];
        }
        float lp;
        const int act = sample_k<NA>(z, legal, u_act, lp);
        a.act_out[2 * e + seat] = (uint8_t)act;
      }
    } else {
      if (!bad && tid < 128 && row < count) {
        float* zo = a.zp_out + ((e * 2 + seat) * 2 + part) * NAP;
#pragma unroll
        for (int o = 0; o < NAP; ++o) zo[o] = zpart[row * NAP + o] + zpart[(128 + row) * NAP + o];
      }
      // a CTA that gave up leaves NaN shares: the next launch stops those envs rather
      // than sample from stale ones (their returns stay those of the state before)
      if (bad && tid < 128 && e >= 0) {
        float* zo = a.zp_out + ((e * 2 + seat) * 2 + part) * NAP;
#pragma unroll
        for (int o = 0; o < NAP; ++o) zo[o] = __int_as_float(0x7FC00000);
      }
    }
    // a tile that gave up wrote no action: its envs stop here, so that no later step of
    // the call applies a stale one
    if (bad && tid < 128 && e >= 0 && owner) a.alive_out[e] = 0;
    if (bad) abort_flag = 1;
  }

  // ---- drain: every MMA and copy of this CTA completes (bounded), free tensor memory ---
  tc::fence_before_sync();
  __syncthreads();
  if (tid == 0 && abort_flag) atomicOr(a.b.status, kStatusTimeout);
  if (warp == 8 && lane == 0) {
    tc::commit(&drain_bar);
    tc::mbar_wait(&drain_bar, 0);
    if (w3_issued) tc::mbar_wait(&w3_bar, 0);
  }
  if (warp == 9 && lane == 0 && abort_flag) {
    // the MMA lane consumed (waited for) every stage unless the CTA aborted; then the
    // copies that may be in flight land before the CTA leaves (bounded waits)
    for (int d = next_chunk - 1; d >= 0 && d >= next_chunk - NST; --d)
      tc::mbar_wait(&full_bar[d % NST], (uint32_t)(d / NST) & 1u);
  }
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 0) {
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, 512);
  }
}

// Test hook: the observation rows this kernel builds (the env's bit-row writer, then the
// constant-1 input at bit obs_dim) for `seat` of every env of a state array (SoA, n envs).
template <class Env>
__global__ void obs_words_kernel(const uint32_t* __restrict__ state, int64_t n, const DevEnv env, int seat,
                                 int words, uint32_t* __restrict__ out) {
  const int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (e >= n) return;
  typename Env::State s;
  load_state(state, n, e, s);
  ObsBits wr{out + e * words, words};
  Env::obs_into(env, s, seat, wr);
  wr.set(env.obs_dim, 1);
}
template <class Env>
cudaError_t launch_obs_words(const uint32_t* state, int64_t n, const DevEnv& env, int seat, int words,
                             uint32_t* out, cudaStream_t s) {
  obs_words_kernel<Env><<<(unsigned)((n + 127) / 128), 128, 0, s>>>(state, n, env, seat, words, out);
  return cudaGetLastError();
}

// Steps after the first are launched with programmatic stream serialization: their CTAs
// may start while the previous step finishes, and the kernel waits (griddepcontrol.wait)
// before it reads or writes anything the previous step touches.  Step 0 follows
// ordinary stream order (its predecessor may be a memset).
template <class Env>
cudaError_t launch_xp_tc(const XpTcArgs& a, int grid, size_t smem, cudaStream_t s) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3(kXpThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  // the two parts of a tile wait on each other: a cluster of two makes them co-resident
  cudaLaunchAttribute attr[2];
  int n = 0;
  if (a.parts == 2) {
    attr[n].id = cudaLaunchAttributeClusterDimension;
    attr[n].val.clusterDim.x = 2;
    attr[n].val.clusterDim.y = 1;
    attr[n].val.clusterDim.z = 1;
    ++n;
  }
  if (a.s > 0) {
    attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[n].val.programmaticStreamSerializationAllowed = 1;
    ++n;
  }
  cfg.attrs = attr;
  cfg.numAttrs = n;
  return cudaLaunchKernelEx(&cfg, xp_tc_kernel<Env>, a);
}

template <class Env>
cudaError_t xp_tc_smem_limit(size_t smem) {
  return cudaFuncSetAttribute(xp_tc_kernel<Env>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
}

}  // namespace aht
