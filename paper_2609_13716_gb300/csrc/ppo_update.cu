// ppo_update.cu -- the PPO ego update (App. C "PPO ego"): the clipped-surrogate loss of
// Schulman et al. 2017 with a clipped value loss and an entropy bonus, its gradient on
// tensor cores, global-norm clipping and Adam (Kingma & Ba 2015), over minibatches of a
// collected trajectory drawn by a keyed permutation.
//
// ppo_grad_kernel: one CTA per SM, each a contiguous run of 64-sample tiles of the
// minibatch.  Per tile the forward (L1, L2 and the output layer as tcgen05 MMAs), the
// per-sample loss gradient, and the backward run in one pass; the weight gradients
// accumulate in tensor memory over the CTA's tiles (dW1 208 columns, dW2 144, dW3^T 16,
// the working accumulator 128: 496 of 512) and leave once, as the CTA's partial sum.  Operands live in shared memory as rows of samples (8 x 16-byte core matrices, 8
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
// Warps w with w % 4 in {0, 1} reach tensor-memory lanes 0..63 (the tile's samples): the 8
// compute warps 0, 1, 4, 5, 8, 9, 12, 13 (four threads per sample, 32 features each).
// Warp 2 issues the MMAs; warps 3, 6, 7 and 10 load the next tile; warp 11 idles.
constexpr int kThreadsPpo = 448;
constexpr int kCompute = 256;
constexpr int kLoaders = 128;
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
constexpr uint32_t kOffSC = kOffPK + kPpoPackedBytes;          // [2][5][64] per-sample scalars
constexpr uint32_t kSmemUsed = kOffSC + 2 * 5 * kRows * 4;
constexpr uint32_t kOffRed = kOffDA2hi;                        // [64][16] f32 end-of-kernel sums
static_assert(kOffH1hi == 26624 && kOffPK == 133120, "layout");
// every M = 128 A operand of a 64-sample buffer reads 64 more rows from what follows
static_assert(kOffX + 2 * kRows * kKP * 2 <= kSmemUsed && kOffDA2lo + 2 * kRows * kH * 2 <= kSmemUsed &&
                  kOffH2lo + 2 * kRows * kH * 2 <= kSmemUsed && kOffDZlo + 2 * kRows * 16 * 2 <= kSmemUsed,
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
  extern __shared__ __align__(16) uint8_t sm[];  // no-swizzle operands need 16 B
  // operands ready (threads -> MMA warp): X, h1, h2, dz, da2, da1
  __shared__ __align__(8) uint64_t opnd_bar[6];
  // products done (commit -> threads): L1, L2, logits, dL/dh2, dL/dh1, dW1 (the tile's last)
  __shared__ __align__(8) uint64_t acc_bar[6];
  __shared__ __align__(8) uint64_t wload_bar, drain_bar;
  __shared__ uint32_t tmem_slot;
  __shared__ volatile int abort_flag;
  enum { kX = 0, kH1 = 1, kH2 = 2, kDZ = 3, kDA2 = 4, kDA1 = 5 };
  enum { kL1 = 0, kL2 = 1, kZ = 2, kDH2 = 3, kDH1 = 4, kDW1 = 5 };

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int n_tiles = (int)(a.B / kRows);
  const int t0 = (int)((int64_t)blockIdx.x * n_tiles / gridDim.x);
  const int t1 = (int)((int64_t)(blockIdx.x + 1) * n_tiles / gridDim.x);
  const int n_it = t1 - t0;
  const uint32_t base = tc::smem_u32(sm);
  const uint8_t* pk = sm + kOffPK;

  if (tid == 0) {
    for (int i = 0; i < 6; ++i) {
      // X: the loader warps; dz: the 64 threads that compute the sample's loss
      tc::mbar_init(&opnd_bar[i], i == kX ? kLoaders : (i == kDZ ? kRows : kCompute));
      tc::mbar_init(&acc_bar[i], 1);
    }
    tc::mbar_init(&wload_bar, 1);
    tc::mbar_init(&drain_bar, 1);
    tc::mbar_init_fence();
    abort_flag = 0;
  }
  if (warp == 0) tc::tmem_alloc(&tmem_slot, 512);
  // constant columns: h1's "ones" feature 128 (carries db2 through dW2) and zero pad; the
  // dz rows' columns 8..15
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
      const uint32_t idZ = tc::idesc_bf16(128, 16);                               // logits
      const uint32_t idH = tc::idesc_bf16(128, kH) | (1u << 16);                  // B MN-major
      const uint32_t id3 = tc::idesc_bf16(128, 16) | (1u << 15) | (1u << 16);     // dW3^T
      const uint32_t id2 = tc::idesc_bf16(128, kH1P) | (1u << 15) | (1u << 16);   // dW2
      const uint32_t id1 = tc::idesc_bf16(128, kKP) | (1u << 15) | (1u << 16);    // dW1
      // descriptors at K-step 0; a K-step adds (its byte stride >> 4) to the address field
      auto kmaj = [&](uint32_t off, int K) { return tc::smem_desc(base + off, 128u, (uint32_t)(K / 8) * 128u); };
      auto mnmaj = [&](uint32_t off, int MN) { return tc::smem_desc(base + off, (uint32_t)(MN / 8) * 128u, 128u); };
      const uint64_t dX = kmaj(kOffX, kKP), dW1 = kmaj(kOffPK + kPkW1, kKP);
      const uint64_t dH1[2] = {kmaj(kOffH1hi, kH1P), kmaj(kOffH1lo, kH1P)};
      const uint64_t dW2 = kmaj(kOffPK + kPkW2, kH), dW2t = mnmaj(kOffPK + kPkW2, kH);
      const uint64_t dH2[2] = {kmaj(kOffH2hi, kH), kmaj(kOffH2lo, kH)};
      const uint64_t dW3[2] = {kmaj(kOffPK + kPkW3hi, kH), kmaj(kOffPK + kPkW3lo, kH)};
      const uint64_t dW3t[2] = {mnmaj(kOffPK + kPkW3hi, kH), mnmaj(kOffPK + kPkW3lo, kH)};
      const uint64_t dDZ[2] = {kmaj(kOffDZhi, 16), kmaj(kOffDZlo, 16)};
      const uint64_t dDA2[2] = {kmaj(kOffDA2hi, kH), kmaj(kOffDA2lo, kH)};
      const uint64_t tDA2[2] = {mnmaj(kOffDA2hi, kH), mnmaj(kOffDA2lo, kH)};
      const uint64_t tH2[2] = {mnmaj(kOffH2hi, kH), mnmaj(kOffH2lo, kH)};  // h2, later dL/da1
      const uint64_t tH1[2] = {mnmaj(kOffH1hi, kH1P), mnmaj(kOffH1lo, kH1P)};
      const uint64_t tDZ[2] = {mnmaj(kOffDZhi, 16), mnmaj(kOffDZlo, 16)};
      const uint64_t tX = mnmaj(kOffX, kKP);
      constexpr uint64_t kS16 = 16;                               // 256 B: 16 features
      constexpr uint64_t kSampK = 2ull * (kH / 8) * 128 >> 4;     // 16 samples of a 128-wide buffer
      constexpr uint64_t kSampK1 = 2ull * (kH1P / 8) * 128 >> 4;  // ... of h1 (144 wide)
      constexpr uint64_t kSampKZ = 2ull * (16 / 8) * 128 >> 4;    // ... of dz (16 wide)
      constexpr uint64_t kSampKX = 2ull * (kKP / 8) * 128 >> 4;   // ... of x (208 wide)
      auto wait_opnd = [&](int i, uint32_t par) {
        if (ok) ok = tc::mbar_wait(&opnd_bar[i], par) && !abort_flag;
        if (ok) tc::fence_after_sync();
        return ok;
      };
      // the three products of a split pair: hi*hi, hi*lo, lo*hi (lo*lo is below 2^-16)
      for (int it = 0; ok && it < n_it; ++it) {
        const uint32_t par = (uint32_t)it & 1u;
        const uint32_t fresh = it == 0 ? 0u : 1u;  // the first tile starts the gradient sums
        // L1: acc = X W1^T (13 K-steps of 16 features)
        if (!wait_opnd(kX, par)) break;
#pragma unroll
        for (int ks = 0; ks < kKP / 16; ++ks)
          tc::mma_ss(tmem + kTmAcc, dX + kS16 * ks, dW1 + kS16 * ks, idL, ks > 0);
        tc::commit(&acc_bar[kL1]);
        // L2: acc = (h1_hi + h1_lo) W2^T
        if (!wait_opnd(kH1, par)) break;
#pragma unroll
        for (int part = 0; part < 2; ++part)
#pragma unroll
          for (int ks = 0; ks < kH / 16; ++ks)
            tc::mma_ss(tmem + kTmAcc, dH1[part] + kS16 * ks, dW2 + kS16 * ks, idL, (part | ks) != 0);
        tc::commit(&acc_bar[kL2]);
        // output layer: acc[0..16) = h2 W3^T
        if (!wait_opnd(kH2, par)) break;
#pragma unroll
        for (int p = 0; p < 3; ++p)
#pragma unroll
          for (int ks = 0; ks < kH / 16; ++ks)
            tc::mma_ss(tmem + kTmAcc, dH2[p == 2 ? 1 : 0] + kS16 * ks, dW3[p == 1 ? 1 : 0] + kS16 * ks, idZ,
                       (p | ks) != 0);
        tc::commit(&acc_bar[kZ]);
        // dL/dh2 = dz W3 into acc, then dW3^T += h2^T dz
        if (!wait_opnd(kDZ, par)) break;
#pragma unroll
        for (int p = 0; p < 3; ++p)
          tc::mma_ss(tmem + kTmAcc, dDZ[p == 2 ? 1 : 0], dW3t[p == 1 ? 1 : 0], idH, p != 0);
        tc::commit(&acc_bar[kDH2]);
#pragma unroll
        for (int p = 0; p < 3; ++p)
#pragma unroll
          for (int ks = 0; ks < kRows / 16; ++ks)
            tc::mma_ss(tmem + kTmDW3, tH2[p == 2 ? 1 : 0] + kSampK * ks, tDZ[p == 1 ? 1 : 0] + kSampKZ * ks,
                       id3, (p | ks) != 0 ? 1u : fresh);
        // dL/dh1 = da2 W2 into acc (its commit also covers dW3: h2's rows may be reused),
        // then dW2 += da2^T [h1 | 1] under epilogue 3
        if (!wait_opnd(kDA2, par)) break;
#pragma unroll
        for (int part = 0; part < 2; ++part)
#pragma unroll
          for (int ks = 0; ks < kH / 16; ++ks)
            tc::mma_ss(tmem + kTmAcc, dDA2[part] + kS16 * ks, dW2t + kSampK * ks, idH, (part | ks) != 0);
        tc::commit(&acc_bar[kDH1]);
#pragma unroll
        for (int p = 0; p < 3; ++p)
#pragma unroll
          for (int ks = 0; ks < kRows / 16; ++ks)
            tc::mma_ss(tmem + kTmDW2, tDA2[p == 2 ? 1 : 0] + kSampK * ks, tH1[p == 1 ? 1 : 0] + kSampK1 * ks,
                       id2, (p | ks) != 0 ? 1u : fresh);
        // dW1 += da1^T [x | 1]
        if (!wait_opnd(kDA1, par)) break;
#pragma unroll
        for (int p = 0; p < 2; ++p)
#pragma unroll
          for (int ks = 0; ks < kRows / 16; ++ks)
            tc::mma_ss(tmem + kTmDW1, tH2[p] + kSampK * ks, tX + kSampKX * ks, id1, (p | ks) != 0 ? 1u : fresh);
        tc::commit(&acc_bar[kDW1]);
      }
      if (!ok) abort_flag = 1;
    }
  } else if (warp == 3 || warp == 6 || warp == 7 || warp == 10) {
    // =============================== loader warps ===================================
    // Loader k (warps 3, 6, 7, 10) owns rows 16k .. 16k + 15 of every tile, two lanes per
    // row (words 26h .. 26h + 25 of the observation row for lane half h): it draws the
    // sample from the permutation and loads its observation words and scalars one tile
    // ahead, into registers; once the previous tile's last MMA has completed it writes
    // them out as the X operand (feature D is the constant 1 that carries db1 through
    // dW1) and the scalar rows, and releases the tile.  The next tile's loads are issued
    // once epilogue 1 is over: the loads slow whatever epilogue they overlap (~1-1.5 K
    // cycles, measured), and epilogue 2 suffers least.
    if (n_it > 0) {
      const int D = a.D, nw = D / 4;
      const int li = warp == 3 ? 0 : (warp == 6 ? 1 : (warp == 7 ? 2 : 3));
      const int row = li * 16 + (lane >> 1), hw = lane & 1;
      constexpr int kHalfWords = kKP / 8;   // 26 words per lane
      const float mu = a.mbstat[0], inv_sd = a.mbstat[1];
      uint32_t ow[kHalfWords];
      float sc[5];
      auto load_tile = [&](int it) {
        const uint32_t j = a.mb * a.B + (uint32_t)(t0 + it) * kRows + (uint32_t)row;
        const uint32_t smp = perm_index(a.key, a.epoch, a.w, a.S, j);
        const uint32_t* orow = reinterpret_cast<const uint32_t*>(a.obs + (size_t)smp * D);
#pragma unroll
        for (int q0 = 0; q0 < kHalfWords; ++q0) {
          const int q = hw * kHalfWords + q0;
          ow[q0] = q < nw ? __ldg(orow + q) : (q == nw ? 1u : 0u);
        }
        if (hw == 0) {
          sc[0] = __int_as_float((int)a.act[smp]);
          sc[1] = a.logp[smp];
          sc[2] = a.val[smp];
          sc[3] = (a.adv[smp] - mu) * inv_sd;
          sc[4] = a.tgt[smp];
        }
      };
      bool ok = true;
      load_tile(0);
      for (int it = 0; it < n_it; ++it) {
        if (it > 0 && ok) ok = tc::mbar_wait(&acc_bar[kDW1], (uint32_t)(it - 1) & 1u);
        ok = __all_sync(0xFFFFFFFFu, ok) && !abort_flag;
        if (!ok) break;
        float* scw = reinterpret_cast<float*>(sm + kOffSC) + (it & 1) * 5 * kRows;
#pragma unroll
        for (int c = 0; c < kHalfWords / 2; ++c)
          *reinterpret_cast<uint4*>(sm + kOffX + canon(row, 8 * (hw * kHalfWords / 2 + c), kKP)) =
              make_uint4(tc::bytes_to_bf16x2(ow[2 * c], 0), tc::bytes_to_bf16x2(ow[2 * c], 2),
                         tc::bytes_to_bf16x2(ow[2 * c + 1], 0), tc::bytes_to_bf16x2(ow[2 * c + 1], 2));
        if (hw == 0) {
#pragma unroll
          for (int k = 0; k < 5; ++k) scw[k * kRows + row] = sc[k];
        }
        tc::fence_proxy_async();
        tc::mbar_arrive(&opnd_bar[kX]);
        if (it + 1 < n_it) {
          if (ok) ok = tc::mbar_wait(&acc_bar[kL2], (uint32_t)it & 1u);  // epilogue 1 is over
          load_tile(it + 1);
        }
      }
      if (!ok) abort_flag = 1;
    }
  } else if ((warp & 2) == 0) {
    // ============================== compute warps ===================================
    const int quarter = warp >> 2;                                 // features 32q .. 32q + 31
    const int row = (warp & 1) * 32 + lane;                       // sample row of the tile
    const int c0 = quarter * 32;
    const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;  // tensor-memory lanes
    const int A = a.n_act;
    const float eps = a.clip_eps, inv_b = 1.0f / (float)a.B;
    const float* b1 = reinterpret_cast<const float*>(pk + kPkB1);
    const float* b2 = reinterpret_cast<const float*>(pk + kPkB2);
    const float* b3 = reinterpret_cast<const float*>(pk + kPkB3);
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
    // tanh(acc + bias) of this thread's 32 columns -> hi | lo bf16 rows at dst (row width W)
    auto act_rows = [&](const float* bias, uint32_t dst_hi, uint32_t dst_lo, int W) {
      uint32_t v[32];
      tc::ld_x32(tmem + kTmAcc + lane_base + c0, v);
      tc::wait_ld();
      uint32_t hi[16], lo[16];
#pragma unroll
      for (int q = 0; q < 16; ++q) {
        const uint64_t x = tc::f2_add(tc::f2_pack(__uint_as_float(v[2 * q]), __uint_as_float(v[2 * q + 1])),
                                      tc::f2_pack(bias[c0 + 2 * q], bias[c0 + 2 * q + 1]));
        tc::split_bf16x2_p(tc::tanh2(x), hi[q], lo[q]);
      }
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        *reinterpret_cast<uint4*>(sm + dst_hi + canon(row, c0 + 8 * q, W)) =
            make_uint4(hi[4 * q], hi[4 * q + 1], hi[4 * q + 2], hi[4 * q + 3]);
        *reinterpret_cast<uint4*>(sm + dst_lo + canon(row, c0 + 8 * q, W)) =
            make_uint4(lo[4 * q], lo[4 * q + 1], lo[4 * q + 2], lo[4 * q + 3]);
      }
    };
    // g (1 - h^2), h = hi + lo from the rows at src (row width W), -> hi | lo rows at dst
    auto grad_rows = [&](uint32_t src_hi, uint32_t src_lo, int W, uint32_t dst_hi, uint32_t dst_lo) {
      uint32_t v[32];
      tc::ld_x32(tmem + kTmAcc + lane_base + c0, v);
      tc::wait_ld();
#pragma unroll
      for (int q8 = 0; q8 < 4; ++q8) {
        const int c = c0 + 8 * q8;
        const uint4 hh = *reinterpret_cast<const uint4*>(sm + src_hi + canon(row, c, W));
        const uint4 hl = *reinterpret_cast<const uint4*>(sm + src_lo + canon(row, c, W));
        const uint32_t hv[4] = {hh.x, hh.y, hh.z, hh.w}, lv4[4] = {hl.x, hl.y, hl.z, hl.w};
        uint32_t dh[4], dl[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          float h0a, h0b, h1a, h1b;
          unpack_bf16x2(hv[q], h0a, h1a);
          unpack_bf16x2(lv4[q], h0b, h1b);
          const uint64_t h = tc::f2_add(tc::f2_pack(h0a, h1a), tc::f2_pack(h0b, h1b));
          const uint64_t one_m = tc::f2_fma(h, tc::f2_sub(0ull, h), tc::f2_pack(1.0f, 1.0f));  // 1 - h^2
          const uint64_t g = tc::f2_pack(__uint_as_float(v[8 * q8 + 2 * q]), __uint_as_float(v[8 * q8 + 2 * q + 1]));
          tc::split_bf16x2_p(tc::f2_mul(g, one_m), dh[q], dl[q]);
        }
        *reinterpret_cast<uint4*>(sm + dst_hi + canon(row, c, kH)) = make_uint4(dh[0], dh[1], dh[2], dh[3]);
        *reinterpret_cast<uint4*>(sm + dst_lo + canon(row, c, kH)) = make_uint4(dl[0], dl[1], dl[2], dl[3]);
      }
    };

    for (int it = 0; it < n_it; ++it) {
      const uint32_t par = (uint32_t)it & 1u;
      // the loader wrote this tile's X and scalars, after the previous tile's last MMA:
      // every operand buffer is free again
      if (!bad && !tc::mbar_wait(&opnd_bar[kX], par)) bad = true;
      if (sync_or()) { bad = true; break; }
      // ---- epilogue 1: h1 = tanh(acc + b1) -> hi | lo rows -------------------------
      wait_acc(kL1, par);
      if (sync_or()) { bad = true; break; }   // every compute thread leaves at the same point
      act_rows(b1, kOffH1hi, kOffH1lo, kH1P);
      release(kH1);
      // ---- epilogue 2: h2 = tanh(acc + b2) -> hi | lo rows -------------------------
      wait_acc(kL2, par);
      if (sync_or()) { bad = true; break; }
      act_rows(b2, kOffH2hi, kOffH2lo, kH);
      release(kH2);
      // ---- the sample's loss and dL/dz (quarter 0, one thread per sample) -----------
      wait_acc(kZ, par);
      if (sync_or()) { bad = true; break; }
      if (quarter == 0) {
        const float* sc = reinterpret_cast<const float*>(sm + kOffSC) + (it & 1) * 5 * kRows;
        const int act = __float_as_int(sc[row]);
        const float lp_old = sc[kRows + row], v_old = sc[2 * kRows + row];
        const float adv_n = sc[3 * kRows + row], ret = sc[4 * kRows + row];
        uint32_t zr[16];
        tc::ld_x16(tmem + kTmAcc + lane_base, zr);
        tc::wait_ld();
        float z[kNO];
#pragma unroll
        for (int o = 0; o < kNO; ++o) z[o] = __uint_as_float(zr[o]) + b3[o];
        // log-softmax, entropy, ratio, clipped surrogate, clipped value loss
        float mx = -FLT_MAX;
#pragma unroll
        for (int o = 0; o < kNO; ++o)
          if (o < A) mx = fmaxf(mx, z[o]);
        float se = 0.f;
#pragma unroll
        for (int o = 0; o < kNO; ++o)
          if (o < A) se += __expf(z[o] - mx);
        const float lse = mx + __logf(se);
        float logp[kNO], prob[kNO], ent = 0.f, lp_a = 0.f;
#pragma unroll
        for (int o = 0; o < kNO; ++o) {
          logp[o] = z[o] - lse;
          prob[o] = o < A ? __expf(logp[o]) : 0.f;
          if (o < A) ent -= prob[o] * logp[o];
          if (o == act) lp_a = logp[o];
        }
        const float rho = __expf(lp_a - lp_old);
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
        const float pg = -fminf(un, cl), lv = 0.5f * fmaxf(u * u, w * w);
        st_loss += pg + a.vf_coef * lv - a.ent_coef * ent;
        st_pg += pg;
        st_v += lv;
        st_ent += ent;
        st_kl += lp_old - lp_a;
        st_clip += fabsf(rho - 1.0f) > eps ? 1.0f : 0.0f;
        uint32_t zh[4], zl[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          dzsum[2 * q] += dz[2 * q];
          dzsum[2 * q + 1] += dz[2 * q + 1];
          split2(dz[2 * q], dz[2 * q + 1], zh[q], zl[q]);
        }
        *reinterpret_cast<uint4*>(sm + kOffDZhi + canon(row, 0, 16)) = make_uint4(zh[0], zh[1], zh[2], zh[3]);
        *reinterpret_cast<uint4*>(sm + kOffDZlo + canon(row, 0, 16)) = make_uint4(zl[0], zl[1], zl[2], zl[3]);
        release(kDZ);
      }
      // ---- dL/da2 = (dz W3) (1 - h2^2) --------------------------------------------
      wait_acc(kDH2, par);
      if (sync_or()) { bad = true; break; }
      grad_rows(kOffH2hi, kOffH2lo, kH, kOffDA2hi, kOffDA2lo);
      release(kDA2);
      // ---- epilogue 3: dL/da1 = (da2 W2) (1 - h1^2) into the h2 rows ----------------
      wait_acc(kDH1, par);
      if (sync_or()) { bad = true; break; }
      grad_rows(kOffH1hi, kOffH1lo, kH1P, kOffH2hi, kOffH2lo);
      release(kDA1);
    }
    if (n_it > 0 && !bad) wait_acc(kDW1, (uint32_t)(n_it - 1) & 1u);  // the last dW1 (all MMAs)
    if (bad) abort_flag = 1;
    // per-CTA sums over the quarter-0 threads: dz (db3) and the loss diagnostics, row order
    __syncwarp();
    tc::bar_or(kComputeBar, kCompute, false);
    float* red = reinterpret_cast<float*>(sm + kOffRed);  // [64][16]
    if (quarter == 0) {
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
#pragma unroll
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
#pragma unroll
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
#pragma unroll
      for (int jj = 0; jj < kNO; ++jj)
        if (jj < A1) part[a.oW3 + (int64_t)jj * kH + o] = n_it == 0 ? 0.f : __uint_as_float(v[jj]);
    }
  }
  if (!abort_flag && tid < 16) {
    const float* red = reinterpret_cast<const float*>(sm + kOffRed);
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

size_t ppo_grad_smem_bytes() { return kSmemUsed; }

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
    // four interleaved fp32 chains (CTA c into chain c % 4), joined in fp64: a fixed order
    // that keeps the dependent-add chain a quarter as long (fp64 adds are slow here)
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
    int c = 0;
    for (; c + 4 <= G; c += 4) {
#pragma unroll
      for (int k = 0; k < 4; ++k) acc[k] += partials[(int64_t)(c + k) * stride + i];
    }
    for (int k = 0; c < G; ++c, ++k) acc[k] += partials[(int64_t)c * stride + i];
    g = ((double)acc[0] + (double)acc[1]) + ((double)acc[2] + (double)acc[3]);
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
    const __nv_bfloat16 hi = __float2bfloat16_rn(p);
    const uint32_t off = tc::canon_offset(jj, k, kH);
    *reinterpret_cast<__nv_bfloat16*>(pk + kPkW3hi + off) = hi;
    *reinterpret_cast<__nv_bfloat16*>(pk + kPkW3lo + off) = __float2bfloat16_rn(p - __bfloat162float(hi));
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
