// aht_common.cuh -- types and device helpers shared by the libaht kernels.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/aht.h"

namespace aht {

constexpr int kThreads = 256;       // threads per CTA of the rollout kernels
constexpr int kMaxPool = 256;       // teammate pool entries passed by value
constexpr int kMaxXpIds = 64;       // ego / teammate ids per cross-play call

// Device status word bits (latched with atomicOr, read by aht_sync).
enum : uint32_t {
  kStatusIllegalAction = 1u,
  kStatusActorMismatch = 2u,
  kStatusBadPolicy = 4u,
  kStatusTimeout = 8u,   // a bounded device wait gave up
  kStatusGrouping = 16u, // a per-episode tile did not find all its envs (tile skipped)
};

// Philox streams (counter word 2).
enum : uint32_t { kStreamAct0 = 0, kStreamAct1 = 1, kStreamReset = 2, kStreamTeammate = 3,
                  kStreamPermute = 4 /* PPO minibatch permutation */,
                  kStreamEpisodeTeammate = 5 /* per-episode teammate draw */ };

struct DevEnv {
  int32_t kind, width, height, n_food, max_level, episode_len, cook_time, soup_reward;
  int32_t obs_dim, n_actions;
};

// Packed fp32 policy: Wt1 [K][H0], b1 [H0], Wt2 [H0][H1], b2 [H1], Wt3 [H1][NOP], b3 [NOP]
// (transposed, so a warp reading one k row of W reads consecutive outputs).
struct MlpDims {
  int32_t K, KP, H0, H1, NA, NOP;
  int64_t stride;  // floats per policy
  int64_t oW1, ob1, oW2, ob2, oW3, ob3;
  // Observations that are a fixed pattern (LBF: every cell word 0x01000000, the open-cell
  // feature set) plus a few changed bytes: the first layer is c + sum over the changed
  // features, c = b1 + W1 x_default kept per policy at oC.
  int32_t sparse;
  int64_t oC;
};
constexpr uint32_t kSparseDefaultWord = 0x01000000u;
constexpr int kSparseCap = 32;  // list entries per row: a count and up to 31 changed features

struct Key {
  uint32_t k0, k1;
};

// ---- Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11) -------------------------------
__device__ __forceinline__ uint4 philox(uint4 c, Key key) {
  uint32_t k0 = key.k0, k1 = key.k1;
#pragma unroll
  for (int i = 0; i < 10; ++i) {
    const uint32_t hi0 = __umulhi(0xD2511F53u, c.x), lo0 = 0xD2511F53u * c.x;
    const uint32_t hi1 = __umulhi(0xCD9E8D57u, c.z), lo1 = 0xCD9E8D57u * c.z;
    c = make_uint4(hi1 ^ c.y ^ k0, lo1, hi0 ^ c.w ^ k1, lo0);
    k0 += 0x9E3779B9u;
    k1 += 0xBB67AE85u;
  }
  return c;
}

// First word of block 0 of (env, step, stream): one draw per action / teammate choice.
__device__ __forceinline__ uint32_t draw0(Key key, uint32_t env, uint32_t step, uint32_t stream) {
  return philox(make_uint4(env, step, stream, 0u), key).x;
}

// Successive draws of one (env, step, stream): draw n is word n % 4 of block n / 4.
struct DrawSeq {
  Key key;
  uint32_t env, step, stream, n;
  uint4 blk;
  __device__ DrawSeq(Key k, uint32_t e, uint32_t t, uint32_t s)
      : key(k), env(e), step(t), stream(s), n(0) {}
  __device__ uint32_t next() {
    const uint32_t w = n & 3u;
    if (w == 0) blk = philox(make_uint4(env, step, stream, n >> 2), key);
    ++n;
    return w == 0 ? blk.x : (w == 1 ? blk.y : (w == 2 ? blk.z : blk.w));
  }
};

// floor(x * n / 2^32)
__device__ __forceinline__ uint32_t uniform_int(uint32_t x, uint32_t n) { return __umulhi(x, n); }
// (x >> 8) * 2^-24, exact in fp32
__device__ __forceinline__ float u01(uint32_t x) {
  return __uint2float_rn(x >> 8) * (1.0f / 16777216.0f);
}

// Observation writers.  The env rules fill a row through clear(), set(k, v) (feature k
// := v), set_bits(k, bits, n) (features k .. k+n-1 := bits 0 .. n-1, n <= 32) and
// set_run(k, n) (features k .. k+n-1 := 1); every feature is written at most once after
// clear(), so a writer that only records ones is exact.
struct ObsBytes {  // one u8 per feature (obs_dim bytes, 4-byte aligned)
  uint8_t* p;
  int words;
  __device__ void clear() {
    uint32_t* w = reinterpret_cast<uint32_t*>(p);
    for (int i = 0; i < words; ++i) w[i] = 0u;
  }
  __device__ void set(int k, uint32_t v) { p[k] = (uint8_t)v; }
  __device__ void set_bits(int k, uint32_t bits, int n) {
    for (int b = 0; b < n; ++b) p[k + b] = (uint8_t)((bits >> b) & 1u);
  }
  __device__ void set_run(int k, int n) {
    for (int b = 0; b < n; ++b) p[k + b] = 1;
  }
};

struct ObsBits {  // one bit per feature of binary observations: bit k % 32 of word k / 32
  uint32_t* w;
  int words;
  __device__ void clear() {
    for (int i = 0; i < words; ++i) w[i] = 0u;
  }
  __device__ void set(int k, uint32_t v) {
    if (v) w[k >> 5] |= 1u << (k & 31);
  }
  __device__ void set_bits(int k, uint32_t bits, int n) {
    if (n < 32) bits &= (1u << n) - 1u;
    if (!bits) return;
    const int s = k & 31;
    w[k >> 5] |= bits << s;
    if (s && s + n > 32) w[(k >> 5) + 1] |= bits >> (32 - s);
  }
  __device__ void set_run(int k, int n) {
    while (n > 0) {
      const int m = n < 32 ? n : 32;
      set_bits(k, m == 32 ? 0xFFFFFFFFu : (1u << m) - 1u, m);
      k += m;
      n -= m;
    }
  }
};

__host__ __device__ constexpr inline int64_t align_up(int64_t x, int64_t a) {
  return (x + a - 1) / a * a;
}

}  // namespace aht
