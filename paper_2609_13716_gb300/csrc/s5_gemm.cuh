// s5_gemm.cuh -- the S5 actor-critic's dense products on tcgen05 tensor cores, with the
// element-wise work that follows each product fused into its epilogue.
//
// C = A B^T per batch member: A [rows][K] activations, B [N][K] weights, both bf16 and
// K-major, fp32 accumulation in tensor memory.  Both operands live in global memory
// already cut into tiles in the canonical no-swizzle K-major layout (core matrix (rb, kb)
// of 8 rows x 8 elements at byte (rb * 8 + kb) * 128 of its tile), so that one 1-D bulk
// copy moves a whole tile into shared memory:
//   activation tile (mt, kt): rows [128 mt, 128 mt + 128) x k [64 kt, 64 kt + 64), 16 KB,
//                             at ((mt * KT + kt) * 16 KB)
//   weight tile (nt, kt):     rows [BN nt, BN nt + BN) x k [64 kt, 64 kt + 64), BN * 128 B,
//                             at ((nt * KT + kt) * BN * 128)
// A persistent kernel walks the output tiles (batch, m-tile, n-tile; n fastest, so that the
// CTAs working on one activation tile at the same time share it in L2, and the weights of
// a layer, a few MB, stay there).  Warp 0 (one lane) streams the stages
// of A and B tiles with bulk copies; warp 1 (one lane) issues the MMAs (M = 128, N = BN,
// K = 16) into one of two tensor-memory accumulators; warps 2-9 read the other one (a
// thread is a row; the warps 2-5 and 6-9 take half of the tile's columns each) and run the
// epilogue, so a tile's epilogue overlaps the next tile's products.
// The epilogues write the next layer's operand directly in the tiled layout:
//   kSplit  v = act(acc + b) as parts bf16 terms (2: hi | lo; 3: hi | lo | hi, the three-
//           term product against [Wh | Wh | Wl]), optionally also fp32 v
//   kSsm    the SSM recurrence x = lbar x_prev + acc (complex, zero before an episode's
//           first step), the state back to global memory and x's [hi | lo | hi] terms
//   kGelu   v = u + gelu(acc + D u) as hi | lo
//   kHeads  h = relu(acc + b) times the output rows: per row and n-tile the partial
//           output sums (a last small kernel adds them in n-tile order)
// Every wait is bounded (2 s); on expiry the kernel records kStatusTimeout, stops,
// drains its MMAs and copies (bounded) and frees tensor memory.
#pragma once
#include "kernels.h"
#include "tc_common.cuh"

namespace aht {
namespace s5g {

constexpr int kBM = 128;          // rows of an output tile (one tensor-memory lane each)
constexpr int kBK = 64;           // k per stage
constexpr int kStages = 4;
constexpr int kThreads = 320;     // producer, MMA, 8 epilogue warps
constexpr int kEpiThreads = 256;
constexpr uint32_t kATile = kBM * kBK * 2;  // 16 KB
constexpr int kMaxOut = 32;       // output rows of the head kernel (actions, or the value)

enum Epi : int { kSplit = 0, kSsm = 1, kGelu = 2, kHeads = 3 };

struct GemmArgs {
  const uint8_t* A;        // tiled activations of batch member 0
  int64_t a_stride;        // bytes between batch members
  const uint8_t* B;        // tiled weights of batch member 0
  int64_t b_stride;
  int32_t m_tiles, n_tiles, k_tiles, batch, BN;
  int64_t n;               // valid rows
  int32_t epi;
  // kSplit: v = act(acc + bias) of output column gc (group g = gc / I, column c = gc % I)
  // goes to matrix (batch + g) of `out` as columns part * I + c, part < parts
  const float* bias;       // [batch][N]
  int32_t relu, parts, I, out_k_tiles;
  uint8_t* out;            // tiled, out_k_tiles tiles of 64 per m-tile
  int64_t out_stride;      // bytes between output matrices
  float* out32;            // optional fp32 copy of v, row-major [n][N] (batch 0)
  // kSsm: acc = [re | im] of P modes (N = 2P, one n-tile)
  const float* lbar;       // [2][P]
  float* state;            // [n][2P]
  const uint8_t* reset;    // [n]
  int32_t P;
  // kGelu
  const float* u;          // [n][N] fp32
  const float* D;          // [N]
  // kHeads: batch member h = head (0 actor, 1 critic); W3 rows of head h: n_out[h] rows
  const float* W3[2];      // [n_out][N] fp32
  int32_t n_out[2];
  float* partial;          // [n][2][n_tiles][2 column halves][kOut slots]
  uint32_t* status;
};

// byte offset of the 16-byte chunk holding row r (of the m-tile), columns [8 kb, 8 kb + 8)
// of k-tile kt, in a tiled activation matrix
__device__ __forceinline__ int64_t chunk_off(int64_t mt, int k_tiles, int kt, int r, int kb) {
  return ((mt * k_tiles + kt) * (int64_t)kATile) + (int64_t)((((r >> 3) << 3) + kb) << 7) + ((r & 7) << 4);
}

// kOut: the widest output count of kHeads (8 or kMaxOut), a compile-time register width.
template <int kOut>
__global__ void __launch_bounds__(kThreads, 1) gemm_kernel(const GemmArgs a) {
  extern __shared__ __align__(16) uint8_t smem[];
  __shared__ __align__(8) uint64_t full_bar[kStages], empty_bar[kStages];
  __shared__ __align__(8) uint64_t accf_bar[2], acce_bar[2], drain_bar;
  __shared__ uint32_t tmem_slot;
  __shared__ volatile int abort_flag;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int BN = a.BN;
  const uint32_t b_tile = (uint32_t)BN * kBK * 2;
  const uint32_t stage_bytes = kATile + b_tile;
  const int n_tiles_total = a.m_tiles * a.n_tiles * a.batch;
  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) {
      tc::mbar_init(&full_bar[s], 1);
      tc::mbar_init(&empty_bar[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      tc::mbar_init(&accf_bar[i], 1);
      tc::mbar_init(&acce_bar[i], kEpiThreads);
    }
    tc::mbar_init(&drain_bar, 1);
    tc::mbar_init_fence();
    abort_flag = 0;
  }
  if (warp == 0) tc::tmem_alloc(&tmem_slot, 512);
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = tmem_slot;
  int issued_stages = 0;  // (producer) stages whose copies were issued

  auto tile_coords = [&](int tile, int& b, int& nt, int& mt) {
    nt = tile % a.n_tiles;
    const int rest = tile / a.n_tiles;
    mt = rest % a.m_tiles;
    b = rest / a.m_tiles;
  };
  auto wait_or_abort = [&](uint64_t* bar, uint32_t parity) {
    bool ok = false;
    for (int tries = 0; tries < 1000 && !ok && !abort_flag; ++tries) ok = tc::mbar_wait(bar, parity, 2000000ull);
    return ok;
  };

  if (warp == 0) {
    // ============================== producer =========================================
    if (lane == 0) {
      int s = 0;
      uint32_t use = 0;  // times stage s was filled before
      bool ok = true;
      for (int tile = blockIdx.x; ok && tile < n_tiles_total; tile += gridDim.x) {
        int b, nt, mt;
        tile_coords(tile, b, nt, mt);
        const uint8_t* A = a.A + b * a.a_stride + (int64_t)mt * a.k_tiles * kATile;
        const uint8_t* B = a.B + b * a.b_stride + (int64_t)nt * a.k_tiles * b_tile;
        for (int kt = 0; kt < a.k_tiles; ++kt) {
          if (use > 0 && !(ok = wait_or_abort(&empty_bar[s], (use - 1) & 1u))) break;
          uint8_t* dst = smem + (size_t)s * stage_bytes;
          tc::mbar_expect_tx(&full_bar[s], stage_bytes);
          tc::bulk_g2s(dst, A + (int64_t)kt * kATile, kATile, &full_bar[s]);
          tc::bulk_g2s(dst + kATile, B + (int64_t)kt * b_tile, b_tile, &full_bar[s]);
          ++issued_stages;
          if (++s == kStages) {
            s = 0;
            ++use;
          }
        }
      }
      if (!ok) abort_flag = 1;
    }
  } else if (warp == 1) {
    // ================================ MMA issue ======================================
    if (lane == 0) {
      const uint32_t idesc = tc::idesc_bf16(kBM, BN);
      int s = 0, j = 0;
      uint32_t fpar = 0;
      bool ok = true;
      const uint32_t base = tc::smem_u32(smem);
      for (int tile = blockIdx.x; ok && tile < n_tiles_total; tile += gridDim.x, ++j) {
        const int acc = j & 1;
        // the epilogue has read this accumulator's previous tile (j - 2)
        if (j >= 2 && !(ok = wait_or_abort(&acce_bar[acc], (uint32_t)((j >> 1) - 1) & 1u))) break;
        tc::fence_after_sync();
        const uint32_t D = tmem + (uint32_t)(acc * 256);
        for (int kt = 0; kt < a.k_tiles; ++kt) {
          if (!(ok = wait_or_abort(&full_bar[s], fpar))) break;
          tc::fence_after_sync();
          const uint32_t sa = base + (uint32_t)s * stage_bytes, sb = sa + kATile;
          const uint64_t da = tc::smem_desc(sa, 128u, 1024u), db = tc::smem_desc(sb, 128u, 1024u);
#pragma unroll
          for (int kk = 0; kk < kBK / 16; ++kk)
            tc::mma_ss(D, da + 16u * kk, db + 16u * kk, idesc, (kt | kk) != 0);
          tc::commit(&empty_bar[s]);  // the stage is free once these products have read it
          if (++s == kStages) {
            s = 0;
            fpar ^= 1u;
          }
        }
        if (ok) tc::commit(&accf_bar[acc]);
      }
      if (!ok) abort_flag = 1;
    }
  } else {
    // ================================ epilogue =======================================
    const int q = warp & 3;                       // tensor-memory lane quadrant
    const int r = 32 * q + lane;                  // row of the tile
    const uint32_t lane_base = (uint32_t)(32 * q) << 16;
    const int ch = (warp - 2) >> 2;               // column half of this warp
    int j = 0;
    bool ok = true;
    for (int tile = blockIdx.x; tile < n_tiles_total; tile += gridDim.x, ++j) {
      int b, nt, mt;
      tile_coords(tile, b, nt, mt);
      const int acc = j & 1;
      bool got = false;
      if (ok) {
        for (int tries = 0; tries < 1000 && !got && !abort_flag; ++tries)
          got = tc::mbar_wait(&accf_bar[acc], (uint32_t)(j >> 1) & 1u, 2000000ull);
      }
      ok = __all_sync(0xFFFFFFFFu, ok && got);  // warp-uniform: tensor-memory loads are collective
      if (!ok) break;
      tc::fence_after_sync();
      const uint32_t T = tmem + (uint32_t)(acc * 256) + lane_base;
      const int64_t row = (int64_t)mt * kBM + r;
      const bool live = row < a.n;
      const int col0 = nt * BN;                   // first output column of the tile
      // this warp's columns: half of the tile's when each half is whole 32-column chunks,
      // else all of them for the first half
      const bool halves = BN % 64 == 0;
      const int cw = halves ? BN / 2 : (ch == 0 ? BN : 0), cbeg = halves ? ch * cw : 0;
      if (a.epi == kSplit) {
        const float* bias = a.bias + (int64_t)b * a.n_tiles * BN;
        for (int c0 = cbeg; c0 < cbeg + cw; c0 += 32) {
          uint32_t v[32];
          tc::ld_x32(T + c0, v);
          tc::wait_ld();
          float x[32];
#pragma unroll
          for (int i = 0; i < 32; i += 4) {
            const float4 bb = __ldg(reinterpret_cast<const float4*>(bias + col0 + c0 + i));
            x[i] = __uint_as_float(v[i]) + bb.x;
            x[i + 1] = __uint_as_float(v[i + 1]) + bb.y;
            x[i + 2] = __uint_as_float(v[i + 2]) + bb.z;
            x[i + 3] = __uint_as_float(v[i + 3]) + bb.w;
          }
          if (a.relu) {
#pragma unroll
            for (int i = 0; i < 32; ++i) x[i] = fmaxf(x[i], 0.0f);
          }
          if (!live) continue;
          if (a.out32) {
            float* o = a.out32 + row * (int64_t)(a.n_tiles * BN) + col0 + c0;
#pragma unroll
            for (int i = 0; i < 32; i += 4) *reinterpret_cast<float4*>(o + i) = make_float4(x[i], x[i + 1], x[i + 2], x[i + 3]);
          }
          const int gc = col0 + c0, g = gc / a.I, c = gc - g * a.I;
          uint8_t* out = a.out + (int64_t)(b + g) * a.out_stride;
          uint32_t hi[16], lo[16];
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            hi[i] = tc::pack_bf16(x[2 * i], x[2 * i + 1]);
            lo[i] = tc::pack_bf16(x[2 * i] - __uint_as_float(hi[i] << 16),
                                  x[2 * i + 1] - __uint_as_float(hi[i] & 0xFFFF0000u));
          }
          for (int part = 0; part < a.parts; ++part) {
            const uint32_t* src = part == 1 ? lo : hi;
            const int oc = part * a.I + c;        // first output column of the 32
#pragma unroll
            for (int k8 = 0; k8 < 4; ++k8) {
              const int col = oc + 8 * k8;
              *reinterpret_cast<uint4*>(out + chunk_off(mt, a.out_k_tiles, col >> 6, r, (col & 63) >> 3)) =
                  make_uint4(src[4 * k8], src[4 * k8 + 1], src[4 * k8 + 2], src[4 * k8 + 3]);
            }
          }
        }
      } else if (a.epi == kSsm) {
        const int P = a.P, pw = P / 2;           // this warp group's modes: [ch pw, ch pw + pw)
        const bool rs = live && a.reset[row] != 0;
        for (int p0 = ch * pw; p0 < ch * pw + pw; p0 += 16) {
          uint32_t vr[16], vi[16];
          tc::ld_x16(T + p0, vr);
          tc::ld_x16(T + P + p0, vi);
          tc::wait_ld();
          if (!live) continue;
          float* st = a.state + row * (int64_t)(2 * P);
          float xr[16], xi[16];
#pragma unroll
          for (int i = 0; i < 16; i += 4) {
            float4 sr = *reinterpret_cast<const float4*>(st + p0 + i);
            float4 si = *reinterpret_cast<const float4*>(st + P + p0 + i);
            if (rs) sr = si = make_float4(0.f, 0.f, 0.f, 0.f);
            const float4 lr = __ldg(reinterpret_cast<const float4*>(a.lbar + p0 + i));
            const float4 li = __ldg(reinterpret_cast<const float4*>(a.lbar + P + p0 + i));
            const float srv[4] = {sr.x, sr.y, sr.z, sr.w}, siv[4] = {si.x, si.y, si.z, si.w};
            const float lrv[4] = {lr.x, lr.y, lr.z, lr.w}, liv[4] = {li.x, li.y, li.z, li.w};
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              xr[i + k] = fmaf(lrv[k], srv[k], fmaf(-liv[k], siv[k], __uint_as_float(vr[i + k])));
              xi[i + k] = fmaf(lrv[k], siv[k], fmaf(liv[k], srv[k], __uint_as_float(vi[i + k])));
            }
            *reinterpret_cast<float4*>(st + p0 + i) = make_float4(xr[i], xr[i + 1], xr[i + 2], xr[i + 3]);
            *reinterpret_cast<float4*>(st + P + p0 + i) = make_float4(xi[i], xi[i + 1], xi[i + 2], xi[i + 3]);
          }
          // [hi | lo | hi] of x = (re | im): parts of 2P columns each
#pragma unroll
          for (int half = 0; half < 2; ++half) {
            const float* x = half ? xi : xr;
            uint32_t hi[8], lo[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) {
              hi[i] = tc::pack_bf16(x[2 * i], x[2 * i + 1]);
              lo[i] = tc::pack_bf16(x[2 * i] - __uint_as_float(hi[i] << 16),
                                    x[2 * i + 1] - __uint_as_float(hi[i] & 0xFFFF0000u));
            }
            for (int part = 0; part < 3; ++part) {
              const uint32_t* src = part == 1 ? lo : hi;
              const int oc = part * 2 * P + half * P + p0;
#pragma unroll
              for (int k8 = 0; k8 < 2; ++k8) {
                const int col = oc + 8 * k8;
                *reinterpret_cast<uint4*>(a.out + chunk_off(mt, a.out_k_tiles, col >> 6, r, (col & 63) >> 3)) =
                    make_uint4(src[4 * k8], src[4 * k8 + 1], src[4 * k8 + 2], src[4 * k8 + 3]);
              }
            }
          }
        }
      } else if (a.epi == kGelu) {
        for (int c0 = cbeg; c0 < cbeg + cw; c0 += 32) {
          uint32_t v[32];
          tc::ld_x32(T + c0, v);
          tc::wait_ld();
          if (!live) continue;
          const int gc = col0 + c0;
          const float* u = a.u + row * (int64_t)(a.n_tiles * BN) + gc;
          float x[32];
#pragma unroll
          for (int i = 0; i < 32; i += 4) {
            const float4 uu = *reinterpret_cast<const float4*>(u + i);
            const float4 dd = __ldg(reinterpret_cast<const float4*>(a.D + gc + i));
            const float uv[4] = {uu.x, uu.y, uu.z, uu.w}, dv[4] = {dd.x, dd.y, dd.z, dd.w};
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              const float y = fmaf(dv[k], uv[k], __uint_as_float(v[i + k]));
              x[i + k] = uv[k] + y * 0.5f * erfcf(-y * 0.70710678118654752f);  // u + gelu(y)
            }
          }
          uint32_t hi[16], lo[16];
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            hi[i] = tc::pack_bf16(x[2 * i], x[2 * i + 1]);
            lo[i] = tc::pack_bf16(x[2 * i] - __uint_as_float(hi[i] << 16),
                                  x[2 * i + 1] - __uint_as_float(hi[i] & 0xFFFF0000u));
          }
          for (int part = 0; part < 2; ++part) {
            const uint32_t* src = part ? lo : hi;
            const int oc = part * a.I + gc;
#pragma unroll
            for (int k8 = 0; k8 < 4; ++k8) {
              const int col = oc + 8 * k8;
              *reinterpret_cast<uint4*>(a.out + chunk_off(mt, a.out_k_tiles, col >> 6, r, (col & 63) >> 3)) =
                  make_uint4(src[4 * k8], src[4 * k8 + 1], src[4 * k8 + 2], src[4 * k8 + 3]);
            }
          }
        }
      } else {  // kHeads
        const float* bias = a.bias + (int64_t)b * a.n_tiles * BN;
        const float* W3 = a.W3[b];
        const int n_out = a.n_out[b];
        const int64_t ldw = (int64_t)a.n_tiles * BN;
        float part[kOut];
#pragma unroll
        for (int o = 0; o < kOut; ++o) part[o] = 0.0f;
        for (int c0 = cbeg; c0 < cbeg + cw; c0 += 32) {
          uint32_t v[32];
          tc::ld_x32(T + c0, v);
          tc::wait_ld();
          const int gc = col0 + c0;
#pragma unroll
          for (int i = 0; i < 32; i += 4) {
            const float4 bb = __ldg(reinterpret_cast<const float4*>(bias + gc + i));
            const float h0 = fmaxf(__uint_as_float(v[i]) + bb.x, 0.0f), h1 = fmaxf(__uint_as_float(v[i + 1]) + bb.y, 0.0f);
            const float h2 = fmaxf(__uint_as_float(v[i + 2]) + bb.z, 0.0f), h3 = fmaxf(__uint_as_float(v[i + 3]) + bb.w, 0.0f);
            // the outputs are independent sums: one chain each, four columns at a time
#pragma unroll
            for (int o = 0; o < kOut; ++o)
              if (o < n_out) {
                const float4 ww = __ldg(reinterpret_cast<const float4*>(W3 + o * ldw + gc + i));
                part[o] = fmaf(h3, ww.w, fmaf(h2, ww.z, fmaf(h1, ww.y, fmaf(h0, ww.x, part[o]))));
              }
          }
        }
        if (live) {
          float* p = a.partial + (((row * 2 + b) * (int64_t)a.n_tiles + nt) * 2 + ch) * kOut;
#pragma unroll
          for (int o = 0; o < kOut; o += 4)
            if (o < n_out) *reinterpret_cast<float4*>(p + o) = make_float4(part[o], part[o + 1], part[o + 2], part[o + 3]);
        }
      }
      tc::fence_before_sync();
      tc::mbar_arrive(&acce_bar[acc]);
    }
    if (!ok) abort_flag = 1;
  }

  // ---- drain: the MMAs and copies this CTA issued complete (bounded), free tensor memory
  tc::fence_before_sync();
  __syncthreads();
  if (tid == 0 && abort_flag) atomicOr(a.status, kStatusTimeout);
  if (warp == 1 && lane == 0) {
    tc::commit(&drain_bar);
    tc::mbar_wait(&drain_bar, 0);
  }
  if (warp == 0 && lane == 0 && abort_flag) {
    // copies still in flight land before the CTA leaves: the last stages issued
    for (int d = issued_stages - 1; d >= 0 && d >= issued_stages - kStages; --d)
      tc::mbar_wait(&full_bar[d % kStages], (uint32_t)(d / kStages) & 1u);
  }
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 0) {
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, 512);
  }
}

inline size_t gemm_smem_bytes(int BN) { return (size_t)kStages * (kATile + (size_t)BN * kBK * 2); }

}  // namespace s5g
}  // namespace aht
