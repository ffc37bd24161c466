// ppo_update.cu -- the PPO ego update (App. C "PPO ego"): the clipped-surrogate loss of
// Schulman et al. 2017 with a clipped value loss and an entropy bonus, its gradient on
// tensor cores, global-norm clipping and Adam (Kingma & Ba 2015), over minibatches of a
// collected trajectory drawn by a keyed permutation.
//
// ppo_grad_kernel: one CTA per SM, each a contiguous run of 64-sample tiles of the
// minibatch.  Per tile the forward (L1, L2 as tcgen05 MMAs, the output layer on CUDA
// cores), the per-sample loss gradient, and the backward run in one pass; the weight
// gradients accumulate in tensor memory over the CTA's tiles (dW1 208 columns, dW2 144,
// dW3^T 16, the working accumulator 128: 496 of 512) and leave once, as the CTA's partial
// sum.  Operands live in shared memory as rows of samples (8 x 16-byte core matrices, 8
// samples x 8 features): the same buffer is the K-major A operand of a forward product
// (samples as M) and the MN-major operand of a weight-gradient product (samples as K).
// Forward products run with M = 128 over a 64-sample tile: the upper 64 rows read the
// next buffer in shared memory and their accumulator lanes are never read.  Activations
// and gradients are split into two bf16 (x = hi + lo, ~2^-17 relative); W1, W2 are bf16.
#include <cfloat>

#include "kernels.h"
#include "tc_common.cuh"

namespace aht {

namespace {

constexpr int kRows = kPpoTile;      // samples per tile
constexpr int kKP = kPpoKP;          // padded input width: obs + the bias column + zeros
constexpr int kH = kPpoHidden;       // hidden width
constexpr int kH1P = 144;            // h1 row width as the B operand of dW2 (+ ones + pad)
constexpr int kNO = 8;               // output rows (actions + value), padded
constexpr int kThreadsPpo = 192;     // warps 0, 1, 4, 5 compute; warp 2 issues MMAs
constexpr int kCompute = 128;
constexpr int kComputeBar = 1;

// shared memory (bytes from the 1024-aligned base)
constexpr uint32_t kOffX = 0;                                  // [64][208] bf16
constexpr uint32_t kOffH1hi = kOffX + kRows * kKP * 2;         // [64][144]
constexpr uint32_t kOffH1lo = kOffH1hi + kRows * kH1P * 2;
constexpr uint32_t kOffDA2hi = kOffH1lo + kRows * kH1P * 2;    // [64][128]
constexpr uint32_t kOffDA2lo = kOffDA2hi + kRows * kH * 2;
constexpr uint32_t kOffH2hi = kOffDA2lo + kRows * kH * 2;      // [64][128]; later dL/da1
constexpr uint32_t kOffH2lo = kOffH2hi + kRows * kH * 2;
constexpr uint32_t kOffDZhi = kOffH2lo + kRows * kH * 2;       // [64][16]
constexpr uint32_t kOffDZlo = kOffDZhi + kRows * 16 * 2;
constexpr uint32_t kOffPK = kOffDZlo + kRows * 16 * 2;         // packed weights
constexpr uint32_t kOffZX = kOffPK + kPpoPackedBytes;          // [2][64][8] f32
constexpr uint32_t kSmemUsed = kOffZX + 2 * kRows * kNO * 4;
static_assert(kOffH1hi == 26624 && kOffPK == 133120, "layout");
// every M = 128 A operand of a 64-sample buffer reads 64 more rows from what follows
static_assert(kOffX + 2 * kRows * kKP * 2 <= kSmemUsed && kOffDA2lo + 2 * kRows * kH * 2 <= kSmemUsed,
              "A operands stay inside shared memory");

// tensor memory columns
constexpr uint32_t kTmAcc = 0, kTmDW1 = 128, kTmDW2 = 336, kTmDW3 = 480;

// ---- minibatch permutation: 4-round Feistel network, cycle-walked below S -------------
__device__ __forceinline__ uint32_t feistel(Key key, uint32_t epoch, int w, uint32_t x) {
  const int rb = w >> 1, lb = w - rb;
  const uint32_t rmask = (uint32_t)((1ull << rb) - 1), lmask = (uint32_t)((1ull << lb) - 1);
  uint32_t L = x >> rb, R = x & rmask;
#pragma unroll
  for (uint32_t r = 0; r < 4; ++r) {
    const uint32_t f = philox(make_uint4((r & 1u) ? L : R, epoch, kStreamPermute, r), key).x;
    if ((r & 1u) == 0) L = (L ^ f) & lmask;
    else R = (R ^ f) & rmask;
  }
  return (L << rb) | R;
}
__device__ __forceinline__ uint32_t perm_index(Key key, uint32_t epoch, int w, uint32_t S, uint32_t x) {
  uint32_t y = x;
  // a cycle of the w-bit permutation through x returns below S within 2^w steps
  for (uint32_t i = 0; i < (1u << w); ++i) {
    y = feistel(key, epoch, w, y);
    if (y < S) break;
  }
  return y < S ? y : x;  // (never taken: keeps every index in range by construction)
}

__device__ __forceinline__ uint32_t canon(int r, int k, int K) { return tc::canon_offset(r, k, K); }

__device__ __forceinline__ void unpack_bf16x2(uint32_t v, float& a, float& b) {
  a = __uint_as_float(v << 16);
  b = __uint_as_float(v & 0xFFFF0000u);
}

// f32 pair (x0, x1) -> hi | lo bf16 pairs
__device__ __forceinline__ void split2(float x0, float x1, uint32_t& hi, uint32_t& lo) {
  tc::split_bf16x2_p(tc::f2_pack(x0, x1), hi, lo);
}

}  // namespace

__global__ void __launch_bounds__(kThreadsPpo, 1) ppo_grad_kernel(const PpoGradArgs a) {
  extern __shared__ __align__(16) uint8_t smem_raw[];
  uint8_t* const sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) uint64_t opnd_bar[4];  // X ready, h1 ready, backward operands, da1
  __shared__ __align__(8) uint64_t acc_bar[4];   // L1, L2, backward products, dW1 done
  __shared__ __align__(8) uint64_t wload_bar, drain_bar;
  __shared__ uint32_t tmem_slot;
  __shared__ volatile int abort_flag;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int n_tiles = (int)(a.B / kRows);
  const int t0 = (int)((int64_t)blockIdx.x * n_tiles / gridDim.x);
  const int t1 = (int)((int64_t)(blockIdx.x + 1) * n_tiles / gridDim.x);
  const int n_it = t1 - t0;
  const uint32_t base = tc::smem_u32(sm);
  const uint8_t* pk = sm + kOffPK;

  if (tid == 0) {
    for (int i = 0; i < 4; ++i) {
      tc::mbar_init(&opnd_bar[i], kCompute);
      tc::mbar_init(&acc_bar[i], 1);
    }
    tc::mbar_init(&wload_bar, 1);
    tc::mbar_init(&drain_bar, 1);
    tc::mbar_init_fence();
    abort_flag = 0;
  }
  if (warp == 0) tc::tmem_alloc(&tmem_slot, 512);
  // constant columns: h1's "ones" feature 128 (carries db2 through dW2), zero pad; dz 8..15
  for (int r = tid; r < kRows; r += blockDim.x) {
    *reinterpret_cast<uint4*>(sm + kOffH1hi + canon(r, 128, kH1P)) = make_uint4(0x3F80u, 0u, 0u, 0u);
    *reinterpret_cast<uint4*>(sm + kOffH1hi + canon(r, 136, kH1P)) = make_uint4(0u, 0u, 0u, 0u);
    *reinterpret_cast<uint4*>(sm + kOffH1lo + canon(r, 128, kH1P)) = make_uint4(0u, 0u, 0u, 0u);
    *reinterpret_cast<uint4*>(sm + kOffH1lo + canon(r, 136, kH1P)) = make_uint4(0u, 0u, 0u, 0u);
    *reinterpret_cast<uint4*>(sm + kOffDZhi + canon(r, 8, 16)) = make_uint4(0u, 0u, 0u, 0u);
    *reinterpret_cast<uint4*>(sm + kOffDZlo + canon(r, 8, 16)) = make_uint4(0u, 0u, 0u, 0u);
  }
  tc::fence_proxy_async();
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = tmem_slot;

  if (warp == 2) {
    // ================================ MMA warp =====================================
    if (lane == 0 && n_it > 0) {
      tc::mbar_expect_tx(&wload_bar, kPpoPackedBytes);
      for (uint32_t off = 0; off < kPpoPackedBytes; off += 32768u)
        tc::bulk_g2s(sm + kOffPK + off, a.packed + off, min(32768u, kPpoPackedBytes - off), &wload_bar);
      bool ok = tc::mbar_wait(&wload_bar, 0);
      const uint32_t idL = tc::idesc_bf16(128, kH);                               // L1, L2
      const uint32_t idH = tc::idesc_bf16(128, kH) | (1u << 16);                  // dh1: B MN-major
      const uint32_t id3 = tc::idesc_bf16(128, 16) | (1u << 15) | (1u << 16);     // dW3^T
      const uint32_t id2 = tc::idesc_bf16(128, kH1P) | (1u << 15) | (1u << 16);   // dW2
      const uint32_t id1 = tc::idesc_bf16(128, kKP) | (1u << 15) | (1u << 16);    // dW1
      const uint32_t pW1 = base + kOffPK + kPkW1, pW2 = base + kOffPK + kPkW2;
      auto wait_opnd = [&](int i, uint32_t par) {
        if (ok) ok = tc::mbar_wait(&opnd_bar[i], par) && !abort_flag;
        if (ok) tc::fence_after_sync();
        return ok;
      };
      for (int it = 0; ok && it < n_it; ++it) {
        const uint32_t par = (uint32_t)it & 1u;
        const bool first = it == 0;
        // L1: acc = X W1^T (13 K-steps of 16 features)
        if (!wait_opnd(0, par)) break;
        for (int ks = 0; ks < kKP / 16; ++ks)
          tc::mma_ss(tmem + kTmAcc, tc::smem_desc(base + kOffX + 256u * ks, 128u, (kKP / 8) * 128u),
                     tc::smem_desc(pW1 + 256u * ks, 128u, (kKP / 8) * 128u), idL, ks > 0);
        tc::commit(&acc_bar[0]);
        // L2: acc = (h1_hi + h1_lo) W2^T
        if (!wait_opnd(1, par)) break;
        for (int part = 0; part < 2; ++part) {
          const uint32_t h1 = base + (part ? kOffH1lo : kOffH1hi);
          for (int ks = 0; ks < kH / 16; ++ks)
            tc::mma_ss(tmem + kTmAcc, tc::smem_desc(h1 + 256u * ks, 128u, (kH1P / 8) * 128u),
                       tc::smem_desc(pW2 + 256u * ks, 128u, (kH / 8) * 128u), idL, (part | ks) != 0);
        }
        tc::commit(&acc_bar[1]);
        // backward: dW3^T += h2^T dz, dW2 += da2^T [h1 | 1], acc = da2 W2 (= dL/dh1)
        if (!wait_opnd(2, par)) break;
        {
          const uint32_t Ah[3] = {kOffH2hi, kOffH2hi, kOffH2lo}, Bz[3] = {kOffDZhi, kOffDZlo, kOffDZhi};
          for (int p = 0; p < 3; ++p)
            for (int ks = 0; ks < kRows / 16; ++ks)
              tc::mma_ss(tmem + kTmDW3, tc::smem_desc(base + Ah[p] + 4096u * ks, 2048u, 128u),
                         tc::smem_desc(base + Bz[p] + 512u * ks, 256u, 128u), id3,
                         !(first && p == 0 && ks == 0));
          const uint32_t Ad[3] = {kOffDA2hi, kOffDA2hi, kOffDA2lo}, Bh[3] = {kOffH1hi, kOffH1lo, kOffH1hi};
          for (int p = 0; p < 3; ++p)
            for (int ks = 0; ks < kRows / 16; ++ks)
              tc::mma_ss(tmem + kTmDW2, tc::smem_desc(base + Ad[p] + 4096u * ks, 2048u, 128u),
                         tc::smem_desc(base + Bh[p] + 4608u * ks, (kH1P / 8) * 128u, 128u), id2,
                         !(first && p == 0 && ks == 0));
          for (int part = 0; part < 2; ++part) {
            const uint32_t da = base + (part ? kOffDA2lo : kOffDA2hi);
            for (int ks = 0; ks < kH / 16; ++ks)
              tc::mma_ss(tmem + kTmAcc, tc::smem_desc(da + 256u * ks, 128u, (kH / 8) * 128u),
                         tc::smem_desc(pW2 + 4096u * ks, 2048u, 128u), idH, (part | ks) != 0);
          }
        }
        tc::commit(&acc_bar[2]);
        // dW1 += da1^T [x | 1]
        if (!wait_opnd(3, par)) break;
        for (int p = 0; p < 2; ++p)
          for (int ks = 0; ks < kRows / 16; ++ks)
            tc::mma_ss(tmem + kTmDW1, tc::smem_desc(base + (p ? kOffH2lo : kOffH2hi) + 4096u * ks, 2048u, 128u),
                       tc::smem_desc(base + kOffX + 6656u * ks, (kKP / 8) * 128u, 128u), id1,
                       !(first && p == 0 && ks == 0));
        tc::commit(&acc_bar[3]);
      }
      if (!ok) abort_flag = 1;
    }
  } else if (warp != 3) {
    // ============================== compute warps ===================================
    const int half = warp >= 4 ? 1 : 0;
    const int row = (warp & 1) * 32 + lane;                       // sample row of the tile
    const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;  // tensor-memory lanes
    const int D = a.D, A = a.n_act;
    const float mu = a.mbstat[0], inv_sd = a.mbstat[1];
    const float eps = a.clip_eps, inv_b = 1.0f / (float)a.B;
    const float* b1 = reinterpret_cast<const float*>(pk + kPkB1);
    const float* b2 = reinterpret_cast<const float*>(pk + kPkB2);
    const float* b3 = reinterpret_cast<const float*>(pk + kPkB3);
    const float* W3 = reinterpret_cast<const float*>(pk + kPkW3);   // [64 pairs][8][2]
    float* ZX = reinterpret_cast<float*>(sm + kOffZX);
    bool bad = n_it > 0 && !tc::mbar_wait(&wload_bar, 0);
    float st_loss = 0.f, st_pg = 0.f, st_v = 0.f, st_ent = 0.f, st_kl = 0.f, st_clip = 0.f;
    float dzsum[kNO] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    auto wait_acc = [&](int i, uint32_t par) {
      if (!bad && !tc::mbar_wait(&acc_bar[i], par)) bad = true;
      bad = __any_sync(0xFFFFFFFFu, bad);
      tc::fence_after_sync();
    };
    auto release = [&](int i) {  // this thread's operand stores are visible to the MMAs
      tc::fence_proxy_async();
      tc::fence_before_sync();
      tc::mbar_arrive(&opnd_bar[i]);
    };
    auto sync_or = [&]() { return tc::bar_or(kComputeBar, kCompute, bad || abort_flag); };

    for (int it = 0; it < n_it; ++it) {
      const uint32_t par = (uint32_t)it & 1u;
      if (it > 0) wait_acc(3, par ^ 1u);        // the previous tile's dW1 read X and da1
      if (sync_or()) { bad = true; break; }
      // ---- gather: sample s of this row, its observation half and scalars ----------
      const uint32_t j = a.mb * a.B + (uint32_t)(t0 + it) * kRows + (uint32_t)row;
      const uint32_t s = perm_index(a.key, a.epoch, a.w, a.S, j);
      {
        const uint32_t* orow = reinterpret_cast<const uint32_t*>(a.obs + (size_t)s * D);
        for (int c = half * 13; c < half * 13 + 13; ++c) {
          uint32_t w2[2];
#pragma unroll
          for (int q = 0; q < 2; ++q) {
            const int f = 8 * c + 4 * q;
            w2[q] = f < D ? __ldg(orow + f / 4) : (f == D ? 1u : 0u);
          }
          const uint4 v = make_uint4(tc::bytes_to_bf16x2(w2[0], 0), tc::bytes_to_bf16x2(w2[0], 2),
                                     tc::bytes_to_bf16x2(w2[1], 0), tc::bytes_to_bf16x2(w2[1], 2));
          *reinterpret_cast<uint4*>(sm + kOffX + canon(row, 8 * c, kKP)) = v;
        }
      }
      const int act = a.act[s];
      const float lp_old = a.logp[s], v_old = a.val[s], ret = a.tgt[s];
      const float adv_n = (a.adv[s] - mu) * inv_sd;
      release(0);
      // ---- epilogue 1: h1 = tanh(acc + b1) -> hi | lo rows -------------------------
      wait_acc(0, par);
      if (sync_or()) { bad = true; break; }   // every compute thread leaves at the same point
      for (int c0 = half * 64; c0 < half * 64 + 64; c0 += 32) {
        uint32_t v[32];
        tc::ld_x32(tmem + kTmAcc + lane_base + c0, v);
        tc::wait_ld();
        uint32_t hi[16], lo[16];
#pragma unroll
        for (int q = 0; q < 16; ++q) {
          const uint64_t x = tc::f2_add(tc::f2_pack(__uint_as_float(v[2 * q]), __uint_as_float(v[2 * q + 1])),
                                        tc::f2_pack(b1[c0 + 2 * q], b1[c0 + 2 * q + 1]));
          tc::split_bf16x2_p(tc::tanh2(x), hi[q], lo[q]);
        }
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          *reinterpret_cast<uint4*>(sm + kOffH1hi + canon(row, c0 + 8 * q, kH1P)) =
              make_uint4(hi[4 * q], hi[4 * q + 1], hi[4 * q + 2], hi[4 * q + 3]);
          *reinterpret_cast<uint4*>(sm + kOffH1lo + canon(row, c0 + 8 * q, kH1P)) =
              make_uint4(lo[4 * q], lo[4 * q + 1], lo[4 * q + 2], lo[4 * q + 3]);
        }
      }
      release(1);
      // ---- epilogue 2: h2, logits, the sample's loss gradient, dL/da2 ---------------
      wait_acc(1, par);
      if (sync_or()) { bad = true; break; }   // every compute thread leaves at the same point
      uint64_t zacc[kNO] = {0, 0, 0, 0, 0, 0, 0, 0};
      for (int c0 = half * 64; c0 < half * 64 + 64; c0 += 32) {
        uint32_t v[32];
        tc::ld_x32(tmem + kTmAcc + lane_base + c0, v);
        tc::wait_ld();
        uint32_t hi[16], lo[16];
#pragma unroll
        for (int q = 0; q < 16; ++q) {
          const uint64_t x = tc::f2_add(tc::f2_pack(__uint_as_float(v[2 * q]), __uint_as_float(v[2 * q + 1])),
                                        tc::f2_pack(b2[c0 + 2 * q], b2[c0 + 2 * q + 1]));
          const uint64_t h = tc::tanh2(x);
          tc::split_bf16x2_p(h, hi[q], lo[q]);
          const ulonglong2* wp = reinterpret_cast<const ulonglong2*>(W3 + (c0 + 2 * q) * kNO);
#pragma unroll
          for (int o = 0; o < kNO; o += 2) {
            const ulonglong2 ww = wp[o / 2];
            zacc[o] = tc::f2_fma(h, ww.x, zacc[o]);
            zacc[o + 1] = tc::f2_fma(h, ww.y, zacc[o + 1]);
          }
        }
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          *reinterpret_cast<uint4*>(sm + kOffH2hi + canon(row, c0 + 8 * q, kH)) =
              make_uint4(hi[4 * q], hi[4 * q + 1], hi[4 * q + 2], hi[4 * q + 3]);
          *reinterpret_cast<uint4*>(sm + kOffH2lo + canon(row, c0 + 8 * q, kH)) =
              make_uint4(lo[4 * q], lo[4 * q + 1], lo[4 * q + 2], lo[4 * q + 3]);
        }
      }
#pragma unroll
      for (int o = 0; o < kNO; ++o) {
        float e0, e1;
        tc::f2_unpack(zacc[o], e0, e1);
        ZX[(half * kRows + row) * kNO + o] = e0 + e1;
      }
      tc::bar_or(kComputeBar, kCompute, false);
      float z[kNO];
#pragma unroll
      for (int o = 0; o < kNO; ++o) z[o] = (ZX[row * kNO + o] + ZX[(kRows + row) * kNO + o]) + b3[o];
      // log-softmax, entropy, ratio, clipped surrogate, clipped value loss
      float mx = -FLT_MAX;
#pragma unroll
      for (int o = 0; o < kNO; ++o)
        if (o < A) mx = fmaxf(mx, z[o]);
      float se = 0.f;
#pragma unroll
      for (int o = 0; o < kNO; ++o)
        if (o < A) se += expf(z[o] - mx);
      const float lse = mx + logf(se);
      float logp[kNO], prob[kNO], ent = 0.f, lp_a = 0.f;
#pragma unroll
      for (int o = 0; o < kNO; ++o) {
        logp[o] = z[o] - lse;
        prob[o] = o < A ? expf(logp[o]) : 0.f;
        if (o < A) ent -= prob[o] * logp[o];
        if (o == act) lp_a = logp[o];
      }
      const float rho = expf(lp_a - lp_old);
      const float rho_c = fminf(fmaxf(rho, 1.0f - eps), 1.0f + eps);
      const float un = rho * adv_n, cl = rho_c * adv_n;
      const float g_rho = un <= cl ? -adv_n : 0.0f;
      float V = 0.f;
#pragma unroll
      for (int o = 0; o < kNO; ++o)
        if (o == A) V = z[o];
      const float vc = v_old + fminf(fmaxf(V - v_old, -eps), eps);
      const float u = V - ret, w = vc - ret;
      const float dV = u * u >= w * w ? u : 0.0f;
      float dz[kNO];
#pragma unroll
      for (int o = 0; o < kNO; ++o) {
        const float pol = g_rho * rho * ((o == act ? 1.0f : 0.0f) - prob[o]) +
                          a.ent_coef * prob[o] * (logp[o] + ent);
        dz[o] = o < A ? pol * inv_b : (o == A ? a.vf_coef * dV * inv_b : 0.0f);
      }
      if (half == 0) {
        const float pg = -fminf(un, cl), lv = 0.5f * fmaxf(u * u, w * w);
        st_loss += pg + a.vf_coef * lv - a.ent_coef * ent;
        st_pg += pg;
        st_v += lv;
        st_ent += ent;
        st_kl += lp_old - lp_a;
        st_clip += fabsf(rho - 1.0f) > eps ? 1.0f : 0.0f;
#pragma unroll
        for (int o = 0; o < kNO; ++o) dzsum[o] += dz[o];
        uint32_t zh[4], zl[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) split2(dz[2 * q], dz[2 * q + 1], zh[q], zl[q]);
        *reinterpret_cast<uint4*>(sm + kOffDZhi + canon(row, 0, 16)) = make_uint4(zh[0], zh[1], zh[2], zh[3]);
        *reinterpret_cast<uint4*>(sm + kOffDZlo + canon(row, 0, 16)) = make_uint4(zl[0], zl[1], zl[2], zl[3]);
      }
      // dL/dh2 = W3^T dz and dL/da2 = dL/dh2 (1 - h2^2) for this half's features
      for (int c0 = half * 64; c0 < half * 64 + 64; c0 += 8) {
        const uint4 hh = *reinterpret_cast<const uint4*>(sm + kOffH2hi + canon(row, c0, kH));
        const uint4 hl = *reinterpret_cast<const uint4*>(sm + kOffH2lo + canon(row, c0, kH));
        const uint32_t hv[4] = {hh.x, hh.y, hh.z, hh.w}, lv4[4] = {hl.x, hl.y, hl.z, hl.w};
        uint32_t dh[4], dl[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int c = c0 + 2 * q;
          const ulonglong2* wp = reinterpret_cast<const ulonglong2*>(W3 + c * kNO);
          uint64_t g = 0;
#pragma unroll
          for (int o = 0; o < kNO; o += 2) {
            const ulonglong2 ww = wp[o / 2];
            g = tc::f2_fma(tc::f2_pack(dz[o], dz[o]), ww.x, g);
            g = tc::f2_fma(tc::f2_pack(dz[o + 1], dz[o + 1]), ww.y, g);
          }
          float h0a, h0b, h1a, h1b;
          unpack_bf16x2(hv[q], h0a, h1a);
          unpack_bf16x2(lv4[q], h0b, h1b);
          const uint64_t h = tc::f2_add(tc::f2_pack(h0a, h1a), tc::f2_pack(h0b, h1b));
          const uint64_t one_m = tc::f2_fma(h, tc::f2_sub(0ull, h), tc::f2_pack(1.0f, 1.0f));  // 1 - h^2
          tc::split_bf16x2_p(tc::f2_mul(g, one_m), dh[q], dl[q]);
        }
        *reinterpret_cast<uint4*>(sm + kOffDA2hi + canon(row, c0, kH)) = make_uint4(dh[0], dh[1], dh[2], dh[3]);
        *reinterpret_cast<uint4*>(sm + kOffDA2lo + canon(row, c0, kH)) = make_uint4(dl[0], dl[1], dl[2], dl[3]);
      }
      release(2);
      // ---- epilogue 3: dL/da1 = (da2 W2) (1 - h1^2) into the h2 buffers --------------
      wait_acc(2, par);
      if (sync_or()) { bad = true; break; }   // every compute thread leaves at the same point
      for (int c0 = half * 64; c0 < half * 64 + 64; c0 += 32) {
        uint32_t v[32];
        tc::ld_x32(tmem + kTmAcc + lane_base + c0, v);
        tc::wait_ld();
#pragma unroll
        for (int q8 = 0; q8 < 4; ++q8) {
          const int c = c0 + 8 * q8;
          const uint4 hh = *reinterpret_cast<const uint4*>(sm + kOffH1hi + canon(row, c, kH1P));
          const uint4 hl = *reinterpret_cast<const uint4*>(sm + kOffH1lo + canon(row, c, kH1P));
          const uint32_t hv[4] = {hh.x, hh.y, hh.z, hh.w}, lv4[4] = {hl.x, hl.y, hl.z, hl.w};
          uint32_t dh[4], dl[4];
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            float h0a, h0b, h1a, h1b;
            unpack_bf16x2(hv[q], h0a, h1a);
            unpack_bf16x2(lv4[q], h0b, h1b);
            const uint64_t h = tc::f2_add(tc::f2_pack(h0a, h1a), tc::f2_pack(h0b, h1b));
            const uint64_t one_m = tc::f2_fma(h, tc::f2_sub(0ull, h), tc::f2_pack(1.0f, 1.0f));
            const uint64_t g = tc::f2_pack(__uint_as_float(v[8 * q8 + 2 * q]), __uint_as_float(v[8 * q8 + 2 * q + 1]));
            tc::split_bf16x2_p(tc::f2_mul(g, one_m), dh[q], dl[q]);
          }
          *reinterpret_cast<uint4*>(sm + kOffH2hi + canon(row, c, kH)) = make_uint4(dh[0], dh[1], dh[2], dh[3]);
          *reinterpret_cast<uint4*>(sm + kOffH2lo + canon(row, c, kH)) = make_uint4(dl[0], dl[1], dl[2], dl[3]);
        }
      }
      release(3);
    }
    if (n_it > 0 && !bad) wait_acc(3, (uint32_t)(n_it - 1) & 1u);  // the last dW1
    if (bad) abort_flag = 1;
    // per-CTA sums of the half-0 rows: dz (db3) and the loss diagnostics, in row order
    __syncwarp();
    tc::bar_or(kComputeBar, kCompute, false);
    float* red = reinterpret_cast<float*>(sm + kOffZX);  // [64][16]
    if (half == 0) {
#pragma unroll
      for (int o = 0; o < kNO; ++o) red[row * 16 + o] = dzsum[o];
      red[row * 16 + 8] = st_loss;
      red[row * 16 + 9] = st_pg;
      red[row * 16 + 10] = st_v;
      red[row * 16 + 11] = st_ent;
      red[row * 16 + 12] = st_kl;
      red[row * 16 + 13] = st_clip;
    }
  }

  // ---- the CTA's partial gradient: tensor-memory rows out, in parameter order ---------
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  float* part = a.partials + (int64_t)blockIdx.x * a.part_stride;
  if (!abort_flag && warp < 4) {
    const int o = warp * 32 + lane;  // tensor-memory lane = output unit (dW1, dW2) / input (dW3^T)
    const uint32_t lb = (uint32_t)(warp * 32) << 16;
    const int D = a.D, A1 = a.n_act + 1;
    for (int c0 = 0; c0 < kKP; c0 += 16) {
      uint32_t v[16];
      tc::ld_x16(tmem + kTmDW1 + lb + c0, v);
      tc::wait_ld();
      for (int k = 0; k < 16; ++k) {
        const int c = c0 + k;
        if (n_it == 0) v[k] = 0u;
        if (c < D) part[a.oW1 + (int64_t)o * D + c] = __uint_as_float(v[k]);
        else if (c == D) part[a.ob1 + o] = __uint_as_float(v[k]);
      }
    }
    for (int c0 = 0; c0 < kH1P; c0 += 16) {
      uint32_t v[16];
      tc::ld_x16(tmem + kTmDW2 + lb + c0, v);
      tc::wait_ld();
      for (int k = 0; k < 16; ++k) {
        const int c = c0 + k;
        if (n_it == 0) v[k] = 0u;
        if (c < kH) part[a.oW2 + (int64_t)o * kH + c] = __uint_as_float(v[k]);
        else if (c == kH) part[a.ob2 + o] = __uint_as_float(v[k]);
      }
    }
    {
      uint32_t v[16];
      tc::ld_x16(tmem + kTmDW3 + lb, v);
      tc::wait_ld();
      for (int jj = 0; jj < A1; ++jj) part[a.oW3 + (int64_t)jj * kH + o] = n_it == 0 ? 0.f : __uint_as_float(v[jj]);
    }
  }
  if (!abort_flag && tid < 16) {
    const float* red = reinterpret_cast<const float*>(sm + kOffZX);
    float acc = 0.f;
    for (int r = 0; r < kRows; ++r) acc += n_it == 0 ? 0.f : red[r * 16 + tid];
    if (tid < a.n_act + 1) part[a.ob3 + tid] = acc;
    if (tid >= 8 && tid < 14) part[a.n_params + (tid - 8)] = acc;
  }

  // ---- drain: every MMA this CTA issued completes (bounded), then free tensor memory ---
  tc::fence_before_sync();
  __syncthreads();
  if (tid == 0 && abort_flag) atomicOr(a.status, kStatusTimeout);
  if (warp == 2 && lane == 0) {
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

size_t ppo_grad_smem_bytes() { return kSmemUsed + 1024; }

cudaError_t ppo_grad_set_smem() {
  return cudaFuncSetAttribute(ppo_grad_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)ppo_grad_smem_bytes());
}

cudaError_t launch_ppo_grad(const PpoGradArgs& a, int grid, cudaStream_t s) {
  ppo_grad_kernel<<<grid, kThreadsPpo, ppo_grad_smem_bytes(), s>>>(a);
  return cudaGetLastError();
}

// ---- per-minibatch advantage mean and 1 / (std + 1e-8) --------------------------------
__global__ void ppo_advstat_kernel(const float* __restrict__ adv, uint32_t S, int w, Key key,
                                   uint32_t epoch0, int M, uint32_t B, double* part) {
  const int mbi = blockIdx.y, e = mbi / M, b = mbi - e * M;
  double s1 = 0.0, s2 = 0.0;
  for (uint32_t j = blockIdx.x * blockDim.x + threadIdx.x; j < B; j += gridDim.x * blockDim.x) {
    const double x = (double)adv[perm_index(key, epoch0 + (uint32_t)e, w, S, (uint32_t)b * B + j)];
    s1 += x;
    s2 += x * x;
  }
  __shared__ double r1[256], r2[256];
  r1[threadIdx.x] = s1;
  r2[threadIdx.x] = s2;
  __syncthreads();
  for (int o = blockDim.x / 2; o > 0; o >>= 1) {
    if ((int)threadIdx.x < o) {
      r1[threadIdx.x] += r1[threadIdx.x + o];
      r2[threadIdx.x] += r2[threadIdx.x + o];
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    part[((int64_t)mbi * gridDim.x + blockIdx.x) * 2] = r1[0];
    part[((int64_t)mbi * gridDim.x + blockIdx.x) * 2 + 1] = r2[0];
  }
}

__global__ void ppo_advstat_final(const double* part, int nb, uint32_t B, int n_mb, float* mbstat) {
  const int mbi = blockIdx.x * blockDim.x + threadIdx.x;
  if (mbi >= n_mb) return;
  double s1 = 0.0, s2 = 0.0;
  for (int k = 0; k < nb; ++k) {
    s1 += part[((int64_t)mbi * nb + k) * 2];
    s2 += part[((int64_t)mbi * nb + k) * 2 + 1];
  }
  const double mu = s1 / B, var = fmax(s2 / B - mu * mu, 0.0);
  mbstat[2 * mbi] = (float)mu;
  mbstat[2 * mbi + 1] = (float)(1.0 / (sqrt(var) + 1e-8));
}

cudaError_t launch_ppo_advstat(const float* adv, uint32_t S, int w, Key key, uint32_t epoch0, int E,
                               int M, uint32_t B, double* part, float* mbstat, cudaStream_t s) {
  ppo_advstat_kernel<<<dim3(kPpoStatBlocks, E * M), 256, 0, s>>>(adv, S, w, key, epoch0, M, B, part);
  ppo_advstat_final<<<(E * M + 63) / 64, 64, 0, s>>>(part, kPpoStatBlocks, B, E * M, mbstat);
  return cudaGetLastError();
}

// ---- sum of the CTAs' partial gradients (fp64, CTA order) and its squared norm --------
__global__ void ppo_reduce_kernel(const float* __restrict__ partials, int G, int64_t stride,
                                  int64_t n_params, double* grad, double* blocksq, float* stats,
                                  float inv_b) {
  const int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  double g = 0.0;
  if (i < n_params) {
    for (int c = 0; c < G; ++c) g += (double)partials[c * stride + i];
    grad[i] = g;
  }
  __shared__ double sq[256];
  sq[threadIdx.x] = i < n_params ? g * g : 0.0;
  __syncthreads();
  for (int o = blockDim.x / 2; o > 0; o >>= 1) {
    if ((int)threadIdx.x < o) sq[threadIdx.x] += sq[threadIdx.x + o];
    __syncthreads();
  }
  if (threadIdx.x == 0) blocksq[blockIdx.x] = sq[0];
  if (blockIdx.x == 0 && threadIdx.x < 6 && stats) {
    double s = 0.0;
    for (int c = 0; c < G; ++c) s += (double)partials[c * stride + n_params + threadIdx.x];
    stats[threadIdx.x] = (float)(s * inv_b);
  }
}

// ---- weights -> the packed block the grad kernel loads -------------------------------
__device__ __forceinline__ void pack_one(const PpoLayout& L, uint8_t* pk, int64_t i, float p) {
  if (i < L.ob1) {
    const int o = (int)(i / L.D), k = (int)(i - (int64_t)o * L.D);
    *reinterpret_cast<__nv_bfloat16*>(pk + kPkW1 + tc::canon_offset(o, k, kKP)) = __float2bfloat16_rn(p);
  } else if (i < L.oW2) {
    reinterpret_cast<float*>(pk + kPkB1)[i - L.ob1] = p;
  } else if (i < L.ob2) {
    const int64_t r = i - L.oW2;
    const int o = (int)(r / kH), k = (int)(r - (int64_t)o * kH);
    *reinterpret_cast<__nv_bfloat16*>(pk + kPkW2 + tc::canon_offset(o, k, kH)) = __float2bfloat16_rn(p);
  } else if (i < L.oW3) {
    reinterpret_cast<float*>(pk + kPkB2)[i - L.ob2] = p;
  } else if (i < L.ob3) {
    const int64_t r = i - L.oW3;
    const int jj = (int)(r / kH), k = (int)(r - (int64_t)jj * kH);
    reinterpret_cast<float*>(pk + kPkW3)[((k >> 1) * kNO + jj) * 2 + (k & 1)] = p;
  } else {
    reinterpret_cast<float*>(pk + kPkB3)[i - L.ob3] = p;
  }
}

__global__ void ppo_pack_kernel(const PpoLayout L, const float* __restrict__ params, uint8_t* pk) {
  const int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (i < L.n_params) pack_one(L, pk, i, params[i]);
}

cudaError_t launch_ppo_pack(const PpoLayout& L, const float* params, uint8_t* pk, cudaStream_t s) {
  ppo_pack_kernel<<<(unsigned)((L.n_params + 255) / 256), 256, 0, s>>>(L, params, pk);
  return cudaGetLastError();
}

// ---- global-norm clipping and Adam, then repack ---------------------------------------
__global__ void ppo_adam_kernel(const PpoAdamArgs a) {
  __shared__ float scale;
  if (threadIdx.x == 0) {
    double s = 0.0;
    for (int b = 0; b < a.n_blocks; ++b) s += a.blocksq[b];
    const double norm = sqrt(s);
    scale = (a.max_grad_norm > 0.f && norm >= (double)a.max_grad_norm) ? (float)((double)a.max_grad_norm / norm) : 1.0f;
  }
  __syncthreads();
  const int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (i >= a.L.n_params) return;
  const float g = (float)a.grad[i] * scale;
  const float m = a.b1 * a.m[i] + (1.0f - a.b1) * g;
  const float v = a.b2 * a.v[i] + (1.0f - a.b2) * g * g;
  const float p = a.params[i] - a.lr * (m / a.c1) / (sqrtf(v / a.c2) + a.eps);
  a.m[i] = m;
  a.v[i] = v;
  a.params[i] = p;
  pack_one(a.L, a.packed, i, p);
}

cudaError_t launch_ppo_reduce_adam(const float* partials, int G, int64_t stride, const PpoAdamArgs& a,
                                   float* stats, float inv_b, bool step, cudaStream_t s) {
  const unsigned nb = (unsigned)((a.L.n_params + 255) / 256);
  ppo_reduce_kernel<<<nb, 256, 0, s>>>(partials, G, stride, a.L.n_params, a.grad, a.blocksq, stats, inv_b);
  if (step) ppo_adam_kernel<<<nb, 256, 0, s>>>(a);
  return cudaGetLastError();
}

__global__ void f64_to_f32_kernel(const double* __restrict__ x, float* __restrict__ y, int64_t n) {
  const int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (i < n) y[i] = (float)x[i];
}

cudaError_t launch_f64_to_f32(const double* x, float* y, int64_t n, cudaStream_t s) {
  f64_to_f32_kernel<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(x, y, n);
  return cudaGetLastError();
}

}  // namespace aht
