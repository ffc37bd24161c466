// mlp_simt.cuh -- fp32 CUDA-core forward of a tile of M policy rows (Sec. 3 policy pi_i).
//
// z = W3 tanh(W2 tanh(W1 o + b1) + b2) + b3 for M rows that share one policy.  The
// observation tile is u8 in shared memory, hidden activations are fp32 in shared
// memory, weights are the packed fp32 (transposed) copy read through L1/L2.  Every
// output is bias + sum_k x_k w_k accumulated with fmaf in increasing k, so a row's
// result does not depend on which tile or slot it occupies.
#pragma once
#include "aht_common.cuh"

namespace aht {

// out[r][c] = act(bias[c] + sum_k in[r][k] * Wt[k][c]) for r < M, c < N, with
// M % 4 == 0, N % 4 == 0, K % 4 == 0.  Each thread owns 4x4 output blocks.
template <bool kInU8, bool kTanh>
__device__ __forceinline__ void dense_tile(const void* __restrict__ in, int in_ld, int M, int K,
                                           const float* __restrict__ Wt,
                                           const float* __restrict__ bias, int N,
                                           float* __restrict__ out, int out_ld) {
  const int ncb = N >> 2;
  const int blocks = (M >> 2) * ncb;
  for (int blk = threadIdx.x; blk < blocks; blk += blockDim.x) {
    const int c0 = (blk % ncb) << 2, r0 = (blk / ncb) << 2;
    const float4 b4 = __ldg(reinterpret_cast<const float4*>(bias + c0));
    float acc[4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      acc[i][0] = b4.x; acc[i][1] = b4.y; acc[i][2] = b4.z; acc[i][3] = b4.w;
    }
    for (int k = 0; k < K; k += 4) {
      float x[4][4];  // [row][kk]
      if (kInU8) {
        const uint8_t* X = static_cast<const uint8_t*>(in);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const uint32_t v = *reinterpret_cast<const uint32_t*>(X + (r0 + i) * in_ld + k);
#pragma unroll
          for (int kk = 0; kk < 4; ++kk) x[i][kk] = (float)((v >> (8 * kk)) & 0xFFu);
        }
      } else {
        const float* H = static_cast<const float*>(in);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const float4 v = *reinterpret_cast<const float4*>(H + (r0 + i) * in_ld + k);
          x[i][0] = v.x; x[i][1] = v.y; x[i][2] = v.z; x[i][3] = v.w;
        }
      }
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        const float4 w = __ldg(reinterpret_cast<const float4*>(Wt + (int64_t)(k + kk) * N + c0));
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          acc[i][0] = fmaf(x[i][kk], w.x, acc[i][0]);
          acc[i][1] = fmaf(x[i][kk], w.y, acc[i][1]);
          acc[i][2] = fmaf(x[i][kk], w.z, acc[i][2]);
          acc[i][3] = fmaf(x[i][kk], w.w, acc[i][3]);
        }
      }
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      float4 o;
      o.x = kTanh ? tanhf(acc[i][0]) : acc[i][0];
      o.y = kTanh ? tanhf(acc[i][1]) : acc[i][1];
      o.z = kTanh ? tanhf(acc[i][2]) : acc[i][2];
      o.w = kTanh ? tanhf(acc[i][3]) : acc[i][3];
      *reinterpret_cast<float4*>(out + (r0 + i) * out_ld + c0) = o;
    }
  }
}

// First layer for m.sparse observations: each row is the default pattern (every word
// kSparseDefaultWord) except a few bytes, so W1 o + b1 = c + sum over the changed
// features f of (o_f - default_f) W1[:, f], with c = b1 + W1 x_default packed per policy.
// One warp per row lists the changed features in increasing order (list[r][0] = count,
// entries (f << 8) | (delta & 0xFF)); then every output adds its row's entries in that
// order, so the result is deterministic.  A row with more changed bytes than the list
// holds (any observation that is not of the pattern) takes the dense sum b1 + W1 o.
// Rows from `live` on are not computed.
__device__ __forceinline__ void sparse_l1_tile(const uint8_t* X, const MlpDims& m, int live,
                                               const float* __restrict__ Wt, const float* __restrict__ b1,
                                               const float* __restrict__ c, uint32_t* list, float* H1) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  const int words = m.K >> 2;
  for (int r = warp; r < live; r += nw) {
    const uint32_t* row = reinterpret_cast<const uint32_t*>(X + r * m.KP);
    uint32_t* L = list + r * kSparseCap;
    int base = 0;
    for (int w0 = 0; w0 < words; w0 += 32) {
      const int wi = w0 + lane;
      const uint32_t v = wi < words ? row[wi] : kSparseDefaultWord;
      int d[4], n = 0;
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        d[kk] = (int)((v >> (8 * kk)) & 0xFFu) - (int)((kSparseDefaultWord >> (8 * kk)) & 0xFFu);
        n += d[kk] != 0;
      }
      int incl = n;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
        if (lane >= o) incl += y;
      }
      int pos = base + incl - n;
#pragma unroll
      for (int kk = 0; kk < 4; ++kk)
        if (d[kk] != 0) {
          if (pos < kSparseCap - 1) L[1 + pos] = ((uint32_t)(4 * wi + kk) << 8) | ((uint32_t)d[kk] & 0xFFu);
          ++pos;
        }
      base += __shfl_sync(0xFFFFFFFFu, incl, 31);
    }
    if (lane == 0) L[0] = (uint32_t)base;
  }
  __syncthreads();
  const int ncb = m.H0 >> 2;
  for (int blk = threadIdx.x; blk < live * ncb; blk += blockDim.x) {
    const int r = blk / ncb, c0 = (blk - r * ncb) << 2;
    const uint32_t* L = list + r * kSparseCap;
    const int n = (int)L[0];
    if (n > kSparseCap - 1) {  // not of the pattern: the dense sum
      float4 acc = __ldg(reinterpret_cast<const float4*>(b1 + c0));
      for (int k = 0; k < m.K; ++k) {
        const float x = (float)X[r * m.KP + k];
        const float4 wv = __ldg(reinterpret_cast<const float4*>(Wt + (int64_t)k * m.H0 + c0));
        acc.x = fmaf(x, wv.x, acc.x);
        acc.y = fmaf(x, wv.y, acc.y);
        acc.z = fmaf(x, wv.z, acc.z);
        acc.w = fmaf(x, wv.w, acc.w);
      }
      *reinterpret_cast<float4*>(H1 + r * m.H0 + c0) =
          make_float4(tanhf(acc.x), tanhf(acc.y), tanhf(acc.z), tanhf(acc.w));
      continue;
    }
    float4 acc = __ldg(reinterpret_cast<const float4*>(c + c0));
    for (int j = 1; j <= n; ++j) {
      const uint32_t e = L[j];
      const float dv = (float)(int8_t)(e & 0xFFu);
      const float4 wv = __ldg(reinterpret_cast<const float4*>(Wt + (int64_t)(e >> 8) * m.H0 + c0));
      acc.x = fmaf(dv, wv.x, acc.x);
      acc.y = fmaf(dv, wv.y, acc.y);
      acc.z = fmaf(dv, wv.z, acc.z);
      acc.w = fmaf(dv, wv.w, acc.w);
    }
    *reinterpret_cast<float4*>(H1 + r * m.H0 + c0) =
        make_float4(tanhf(acc.x), tanhf(acc.y), tanhf(acc.z), tanhf(acc.w));
  }
}

// Whole policy forward for an M-row tile: X u8 [M][KP] -> Z f32 [M][NOP].  list: the
// sparse first layer's scratch (M * kSparseCap words; unused unless m.sparse), which
// computes rows < live only (the others' outputs are then undefined).
// Synchronises the CTA between layers and at the end.
__device__ __forceinline__ void mlp_tile(const float* __restrict__ w, const MlpDims& m,
                                         const uint8_t* X, float* H1, float* H2, float* Z,
                                         int M, uint32_t* list, int live) {
  if (m.sparse)
    sparse_l1_tile(X, m, live, w + m.oW1, w + m.ob1, w + m.oC, list, H1);
  else
    dense_tile<true, true>(X, m.KP, M, m.K, w + m.oW1, w + m.ob1, m.H0, H1, m.H0);
  __syncthreads();
  dense_tile<false, true>(H1, m.H0, M, m.H0, w + m.oW2, w + m.ob2, m.H1, H2, m.H1);
  __syncthreads();
  dense_tile<false, false>(H2, m.H1, M, m.H1, w + m.oW3, w + m.ob3, m.NOP, Z, m.NOP);
  __syncthreads();
}

// Masked categorical inverse-CDF sample in fp32: a = min{k : u*Z < S_k} over the legal
// actions (S_k = sum_{j<=k} exp(z_j - max)), else the last legal action.
__device__ __forceinline__ int sample_row(const float* z, int K, uint32_t legal, float u,
                                          float& logp) {
  float m = -INFINITY;
  for (int k = 0; k < K; ++k)
    if ((legal >> k) & 1u) m = fmaxf(m, z[k]);
  float S[24];
  float run = 0.0f;
  for (int k = 0; k < K; ++k) {
    if ((legal >> k) & 1u) run = __fadd_rn(run, expf(z[k] - m));
    S[k] = run;
  }
  const float target = u * run;
  int a = -1;
  for (int k = 0; k < K; ++k)
    if (a < 0 && target < S[k]) a = k;
  if (a < 0)
    for (int k = K - 1; k >= 0; --k)
      if (a < 0 && ((legal >> k) & 1u)) a = k;
  logp = z[a] - m - logf(run);
  return a;
}

// The same sample for a compile-time action count, all in registers.
template <int K, int N>
__device__ __forceinline__ int sample_k(const float (&z)[N], uint32_t legal, float u, float& logp) {
  static_assert(K <= N, "logit array shorter than the action count");
  float m = -INFINITY;
#pragma unroll
  for (int k = 0; k < K; ++k)
    if ((legal >> k) & 1u) m = fmaxf(m, z[k]);
  float S[K];
  float run = 0.0f;
#pragma unroll
  for (int k = 0; k < K; ++k) {
    if ((legal >> k) & 1u) run = __fadd_rn(run, expf(z[k] - m));
    S[k] = run;
  }
  const float target = u * run;
  int a = -1;
#pragma unroll
  for (int k = K - 1; k >= 0; --k)
    if (target < S[k]) a = k;
  if (a < 0) {
#pragma unroll
    for (int k = 0; k < K; ++k)
      if ((legal >> k) & 1u) a = k;
  }
  float za = z[0];
#pragma unroll
  for (int k = 1; k < K; ++k)
    if (a == k) za = z[k];
  logp = za - m - logf(run);
  return a;
}

}  // namespace aht
