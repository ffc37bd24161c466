// aht_api.cu -- the C ABI of libaht.so (declared in include/aht.h): argument checks,
// context memory, weight packing and kernel launches.  No compute happens on the host
// except packing the population once in aht_create.
#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <string>
#include <vector>

#include "kernels.h"
#include "rollout_impl.cuh"
#include "tc_common.cuh"

using namespace aht;

namespace {

thread_local std::string g_err;

aht_status fail(aht_status s, const std::string& msg) {
  g_err = msg;
  return s;
}

#define AHT_CUDA(call)                                                                   \
  do {                                                                                   \
    cudaError_t e_ = (call);                                                             \
    if (e_ != cudaSuccess)                                                               \
      return fail(AHT_ECUDA, std::string(#call) + ": " + cudaGetErrorString(e_));        \
  } while (0)

// Device and pinned allocations of contexts go through these: they count the blocks a
// context holds (aht_debug_live_allocs) and let a test make the n-th allocation fail
// (aht_debug_fail_alloc) without touching the device.
std::atomic<int64_t> g_fail_countdown{0};  // > 0: the allocation that brings it to 0 fails
std::atomic<int64_t> g_live_allocs{0};
bool alloc_hook_fires() {
  int64_t n = g_fail_countdown.load();
  while (n > 0 && !g_fail_countdown.compare_exchange_weak(n, n - 1)) {
  }
  return n == 1;
}
cudaError_t ctx_malloc(void** p, size_t bytes) {
  if (alloc_hook_fires()) return cudaErrorMemoryAllocation;
  const cudaError_t e = cudaMalloc(p, bytes);
  if (e == cudaSuccess) ++g_live_allocs;
  return e;
}
cudaError_t ctx_malloc_host(void** p, size_t bytes) {
  if (alloc_hook_fires()) return cudaErrorMemoryAllocation;
  const cudaError_t e = cudaMallocHost(p, bytes);
  if (e == cudaSuccess) ++g_live_allocs;
  return e;
}
void ctx_free(void* p) {
  if (p && cudaFree(p) == cudaSuccess) --g_live_allocs;
}
void ctx_free_host(void* p) {
  if (p && cudaFreeHost(p) == cudaSuccess) --g_live_allocs;
}

struct DeviceGuard {
  int prev = -1;
  explicit DeviceGuard(int dev) {
    if (cudaGetDevice(&prev) == cudaSuccess && prev != dev) cudaSetDevice(dev);
    else prev = -1;
  }
  ~DeviceGuard() {
    if (prev >= 0) cudaSetDevice(prev);
  }
};

struct EnvOps {
  cudaError_t (*ppo)(const PpoArgs&, int, size_t, cudaStream_t);
  cudaError_t (*xplay)(const XpArgs&, int, size_t, cudaStream_t);
  cudaError_t (*forced)(const ForcedArgs&, cudaStream_t);
  cudaError_t (*reset)(const ResetArgs&, cudaStream_t);
  int (*words)();
  int (*bytes)();
  cudaError_t (*smem_limit)(size_t);
  int max_rows;  // largest tile that fits the hidden activations of typical sizes
  int (*occupancy)(int which, size_t smem);  // resident CTAs per SM of the CUDA-core kernels
};

EnvOps ops_for(int kind) {
  switch (kind) {
    case AHT_LBF:
      return {lbf_ppo, lbf_xplay, lbf_forced, lbf_reset, lbf_state_words, lbf_state_bytes, lbf_set_smem_limit,
              128, lbf_occupancy};
    case AHT_OVERCOOKED:
      return {overcooked_ppo, overcooked_xplay, overcooked_forced, overcooked_reset,
              overcooked_state_words, overcooked_state_bytes, overcooked_set_smem_limit, 64,
              overcooked_occupancy};
    case AHT_MINI_HANABI:
      return {minihanabi_ppo, minihanabi_xplay, minihanabi_forced, minihanabi_reset,
              minihanabi_state_words, minihanabi_state_bytes, minihanabi_set_smem_limit, 64,
              minihanabi_occupancy};
    default:
      return {hanabi_ppo, hanabi_xplay, hanabi_forced, hanabi_reset, hanabi_state_words,
              hanabi_state_bytes, hanabi_set_smem_limit, 32, hanabi_occupancy};
  }
}

constexpr uint32_t kStateMagic = 0x31544841u;  // "AHT1"

struct StateHeader {
  uint32_t magic, kind, n_words, pad;
  int64_t n_envs;
  uint64_t seed;
  int64_t step;
};

}  // namespace

struct aht_ctx {
  int device = 0;
  cudaStream_t stream = nullptr;
  aht_env_desc desc{};
  DevEnv env{};
  MlpDims mlp{};
  EnvOps ops{};
  int32_t n_policies = 0;
  int64_t n_envs = 0;
  uint64_t seed = 0;
  int64_t step = 0;
  size_t smem_optin = 0;
  int n_sms = 0;
  int64_t max_tiles = 0;
  // device memory, all allocated in aht_create
  uint32_t* state = nullptr;
  float* weights = nullptr;
  int32_t* perm = nullptr;
  int4* tiles = nullptr;
  float* xp_returns = nullptr;
  float* last_value = nullptr;
  uint32_t* ep_step = nullptr;  // [n_envs] step each env's current episode began
  uint8_t* rs_kidx = nullptr;   // [2][align_up(n_envs, 16)] per-episode pool index by step parity
  int32_t* rs_hist = nullptr;   // [3][kMaxPool] envs per pool index, by step mod 3
  uint32_t* status = nullptr;
  // test hook (aht_debug_logits): caller-owned output buffer of the tensor-core kernels
  float* dbg_logits = nullptr;
  int64_t dbg_floats = 0;
  // failure-detection hook (aht_debug_expire_at): one tensor-core call waits in vain
  int32_t dbg_expire_step = -1;
  uint64_t dbg_expire_ns = 0;
  // tensor-core path (bf16 LBF populations that fit shared and tensor memory)
  int32_t weight_dtype = AHT_BF16;
  bool tc = false;
  TcDims tcd{};
  uint8_t* tcw = nullptr;
  size_t tc_smem = 0;
  uint8_t* tc_staging = nullptr;
  // streamed tensor-core cross-play (bf16 Overcooked / Hanabi populations of width 256/512)
  bool wide = false;
  WideDims wd{};
  uint8_t* wtcw = nullptr;
  uint8_t* wide_staging = nullptr;  // pinned, one streamed block (aht_set_policy)
  size_t wide_smem = 0;
  uint32_t* xp_st[2] = {};
  uint8_t* xp_act[2] = {};
  float* xp_zp[2] = {};
  uint8_t* xp_alive[2] = {};
  int32_t* xp_nsteps = nullptr;
  // two-part tiles (H = 512): the parts' exchange slots and flags, and the launch stamp
  uint8_t* xp_xch = nullptr;
  uint32_t* xp_xflag = nullptr;
  int64_t xp_slots = 0;
  uint32_t xp_stamp = 0;
  // pinned host staging for aht_set_policy, and the event pool of the kernel timer
  float* staging = nullptr;
  cudaEvent_t upload_done = nullptr;
  static constexpr int kTimerPairs = 256;
  cudaEvent_t ev[2 * kTimerPairs] = {};
  bool timing = false;
  int n_pending = 0;
  double timed_ms = 0.0;
  int64_t timed_launches = 0;
};

namespace {

Batch batch_of(const aht_ctx* c) {
  Batch b;
  b.env = c->env;
  b.mlp = c->mlp;
  b.weights = c->weights;
  b.key = Key{(uint32_t)(c->seed & 0xFFFFFFFFu), (uint32_t)(c->seed >> 32)};
  b.status = c->status;
  return b;
}

aht_status check_env(const aht_env_desc* d, DevEnv* out) {
  if (!d) return fail(AHT_EINVAL, "env desc is NULL");
  DevEnv e{};
  e.kind = d->kind;
  e.width = d->width;
  e.height = d->height;
  e.n_food = d->n_food;
  e.max_level = d->max_agent_level;
  e.episode_len = d->episode_len;
  e.cook_time = d->cook_time;
  e.soup_reward = d->soup_reward;
  if (d->kind == AHT_LBF) {
    if (d->width < 3 || d->width > 12 || d->height < 3 || d->height > 12)
      return fail(AHT_EINVAL, "LBF width/height must be in 3..12");
    if (d->n_food < 1 || d->n_food > 3) return fail(AHT_EINVAL, "LBF n_food must be in 1..3");
    if (d->max_agent_level < 1 || d->max_agent_level > 9)
      return fail(AHT_EINVAL, "LBF max_agent_level must be in 1..9");
    if (d->episode_len < 1) return fail(AHT_EINVAL, "LBF episode_len must be >= 1");
    e.obs_dim = d->width * d->height * 4;
    e.n_actions = 6;
  } else if (d->kind == AHT_OVERCOOKED) {
    if (d->width != 5 || d->height != 4) return fail(AHT_EINVAL, "Overcooked kitchen is 5x4");
    if (d->episode_len < 1) return fail(AHT_EINVAL, "Overcooked episode_len must be >= 1");
    if (d->cook_time < 0 || d->cook_time > 255) return fail(AHT_EINVAL, "cook_time must be in 0..255");
    e.obs_dim = 520;
    e.n_actions = 6;
  } else if (d->kind == AHT_HANABI) {
    if (d->episode_len != 0) return fail(AHT_EINVAL, "Hanabi episode_len must be 0 (to termination)");
    e.obs_dim = 660;
    e.n_actions = 20;
  } else if (d->kind == AHT_MINI_HANABI) {
    if (d->episode_len != 0) return fail(AHT_EINVAL, "Mini Hanabi episode_len must be 0 (to termination)");
    e.obs_dim = 156;
    e.n_actions = 10;
  } else {
    return fail(AHT_EINVAL, "unknown env kind");
  }
  *out = e;
  return AHT_OK;
}

MlpDims make_dims(int K, int H0, int H1, int NA, bool sparse) {
  MlpDims m{};
  m.K = K;
  m.KP = (int)align_up(K, 16);
  m.H0 = H0;
  m.H1 = H1;
  m.NA = NA;
  m.NOP = (int)align_up(NA + 1, 4);
  int64_t o = 0;
  m.oW1 = o; o += (int64_t)K * H0;
  m.ob1 = o; o += H0;
  m.oW2 = o; o += (int64_t)H0 * H1;
  m.ob2 = o; o += H1;
  m.oW3 = o; o += (int64_t)H1 * m.NOP;
  m.ob3 = o; o += m.NOP;
  m.sparse = sparse ? 1 : 0;
  m.oC = o; o += sparse ? H0 : 0;
  m.stride = align_up(o, 4);
  return m;
}

float to_f32(const void* p, int64_t i, int dtype) {
  if (dtype == AHT_FP32) return static_cast<const float*>(p)[i];
  uint32_t bits = (uint32_t) static_cast<const uint16_t*>(p)[i] << 16;
  float f;
  std::memcpy(&f, &bits, 4);
  return f;
}

// Packs one policy into dst (m.stride floats): fp32, transposed [in][out], the last layer
// padded to NOP columns (column n_actions is the value row when present, else zero).
aht_status pack_policy(const MlpDims& m, const void* const* W, const void* const* b, int dtype,
                       int vh, float* dst) {
  if (vh != 0 && vh != 1) return fail(AHT_EINVAL, "has_value_head entries must be 0 or 1");
  if (dtype != AHT_FP32 && dtype != AHT_BF16) return fail(AHT_EINVAL, "weight_dtype must be AHT_FP32 or AHT_BF16");
  const int esz = dtype == AHT_FP32 ? 4 : 2;
  const int ins[3] = {m.K, m.H0, m.H1};
  const int outs[3] = {m.H0, m.H1, m.NA + vh};
  const int64_t oW[3] = {m.oW1, m.oW2, m.oW3}, ob[3] = {m.ob1, m.ob2, m.ob3};
  const int cols[3] = {m.H0, m.H1, m.NOP};
  std::fill(dst, dst + m.stride, 0.0f);
  std::vector<uint8_t> tmp;
  // Host memory (pageable or pinned) is read in place; device memory is copied first.
  auto host_view = [&](const void* p, size_t bytes, const void** out) -> bool {
    cudaPointerAttributes at{};
    if (cudaPointerGetAttributes(&at, p) != cudaSuccess) cudaGetLastError();
    if (at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged) {
      tmp.resize(bytes);
      if (cudaMemcpy(tmp.data(), p, bytes, cudaMemcpyDeviceToHost) != cudaSuccess) return false;
      *out = tmp.data();
    } else {
      *out = p;
    }
    return true;
  };
  for (int l = 0; l < 3; ++l) {
    if (!W[l] || !b[l]) return fail(AHT_EINVAL, "NULL weight pointer");
    const void* src = nullptr;
    if (!host_view(W[l], (size_t)outs[l] * ins[l] * esz, &src)) return fail(AHT_ECUDA, "copying weights failed");
    for (int n = 0; n < outs[l]; ++n)
      for (int k = 0; k < ins[l]; ++k)
        dst[oW[l] + (int64_t)k * cols[l] + n] = to_f32(src, (int64_t)n * ins[l] + k, dtype);
    if (!host_view(b[l], (size_t)outs[l] * esz, &src)) return fail(AHT_ECUDA, "copying biases failed");
    for (int n = 0; n < outs[l]; ++n) dst[ob[l] + n] = to_f32(src, n, dtype);
  }
  if (m.sparse) {  // c = b1 + W1 x_default in fp64, rounded once
    for (int n = 0; n < m.H0; ++n) {
      double acc = dst[m.ob1 + n];
      for (int w = 0; w < m.K / 4; ++w)
        for (int kk = 0; kk < 4; ++kk) {
          const uint32_t x = (kSparseDefaultWord >> (8 * kk)) & 0xFFu;
          if (x) acc += (double)x * dst[m.oW1 + (int64_t)(4 * w + kk) * m.H0 + n];
        }
      dst[m.oC + n] = (float)acc;
    }
  }
  return AHT_OK;
}

// Tensor-core block layout of one policy (see TcDims); fp32 populations get the bf16
// remainder copies of W1 and W2.
TcDims make_tc_dims(const MlpDims& m, bool split) {
  TcDims t{};
  t.KP = (int)align_up(m.K + 1, 16);
  t.H0 = m.H0;
  t.H1 = m.H1;
  t.split = split ? 1 : 0;
  // an observation wider than an agent's 256 A-operand columns: the first layer runs on
  // CUDA cores from the observation's changed features (LBF), W1 stays out of the block
  t.sparse = (m.sparse && t.KP > 256) ? 1 : 0;
  const uint32_t w1 = t.sparse ? 0u : (uint32_t)(m.H0 * t.KP * 2);
  uint32_t o = 0;
  t.oW1 = o; o += w1;
  t.oW2 = o; o += (uint32_t)(m.H1 * m.H0 * 2);
  if (split) {
    t.oW1lo = o; o += w1;
    t.oW2lo = o; o += (uint32_t)(m.H1 * m.H0 * 2);
  }
  t.oW3 = o; o += (uint32_t)(m.H1 * 8 * 4);
  t.ob2 = o; o += (uint32_t)(m.H1 * 4);
  t.ob3 = o; o += 8 * 4;
  t.pol_bytes = (uint32_t)align_up(o, 16);
  return t;
}

// Shared memory of the tensor-core kernel: both policies' blocks, the u8 observation
// tile [128][obs_dim], 128 env states, 128 teammate actions and the output layer's
// partial sums [2 agents][2 halves][128][8] fp32.
size_t tc_smem_bytes(const TcDims& t, int obs_dim, int state_bytes) {
  return 2 * (size_t)t.pol_bytes + align_up(128 * obs_dim, 16) + align_up(128 * state_bytes, 16) + 128 +
         4 * 128 * 8 * 4;
}

// The tensor-core path applies to LBF populations whose padded observation (KP/2
// columns) and hidden layers (<= 128 columns each, multiples of 64) fit the 256
// tensor-memory columns each agent uses, and whose two policy blocks fit shared memory
// (fp32 populations hold each weight as a bf16 pair, twice the bytes).
bool tc_eligible(const aht_ctx* c, int dtype) {
  const MlpDims& m = c->mlp;
  if (c->env.kind != AHT_LBF) return false;
  const TcDims t = make_tc_dims(m, dtype == AHT_FP32);
  if ((t.KP > 256 && !t.sparse) || m.H0 > 128 || m.H1 > 128 || m.H0 % 64 || m.H1 % 64 || m.NA + 1 > 8)
    return false;
  return m.K % 4 == 0 && tc_smem_bytes(t, m.K, c->ops.bytes()) <= c->smem_optin;
}

// Streamed tensor-core block of a wide policy (see WideDims).
WideDims make_wide_dims(const MlpDims& m) {
  WideDims w{};
  w.KP = (int)align_up(m.K + 1, 16);
  w.H = m.H0;
  w.NAP = (int)align_up(m.NA, 4);
  w.n_l1 = (w.H / 256) * (w.KP / 16);
  w.n_l2 = (w.H / 256) * (w.H / 16);
  uint32_t o = (uint32_t)(w.n_l1 + w.n_l2) * kWideChunk;
  // W3 as bf16 B fragments of mma.sync m16n8k16: [H / 16 unit chunks][n-tiles of 8
  // outputs][32 threads][2 words]
  w.oW3 = o; o += (uint32_t)(w.H / 16) * (uint32_t)((w.NAP + 7) / 8) * 256u;
  w.ob2 = o; o += (uint32_t)(w.H * 4);
  w.ob3 = o; o += (uint32_t)(w.NAP * 4);
  w.pol_bytes = (uint32_t)align_up(o, 1024);
  return w;
}

// Binary-observation games with bf16 weights and equal hidden widths of 256 or 512 run
// their cross-play steps on the streamed tensor-core kernel.
bool wide_eligible(const aht_ctx* c, int dtype) {
  const MlpDims& m = c->mlp;
  if (dtype != AHT_BF16 || c->env.kind == AHT_LBF) return false;
  if (m.H0 != m.H1 || (m.H0 != 256 && m.H0 != 512)) return false;
  // the 128 env states of a tile live at the start of the operand region during the transition
  if (128 * (size_t)c->ops.bytes() > xp_tc_state_bytes(make_wide_dims(m))) return false;
  return xp_tc_smem_bytes(make_wide_dims(m)) <= c->smem_optin;
}

bool read_host(const void* p, size_t bytes, std::vector<uint8_t>& tmp, const void** out) {
  cudaPointerAttributes at{};
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) cudaGetLastError();
  if (at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged) {
    tmp.resize(bytes);
    if (cudaMemcpy(tmp.data(), p, bytes, cudaMemcpyDeviceToHost) != cudaSuccess) return false;
    *out = tmp.data();
  } else {
    *out = p;
  }
  return true;
}

// Nearest-even bf16 of an fp32 value (bits), and the fp32 value of bf16 bits.
uint16_t bf16_rne(float f) {
  uint32_t u;
  std::memcpy(&u, &f, 4);
  return (uint16_t)((u + 0x7FFFu + ((u >> 16) & 1u)) >> 16);
}
float bf16_val(uint16_t h) {
  const uint32_t u = (uint32_t)h << 16;
  float f;
  std::memcpy(&f, &u, 4);
  return f;
}

// Packs one policy into its tensor-core block (dst: t.pol_bytes bytes).  bf16 weights go
// in as they are; fp32 weights w as hi = bf16(w) and lo = bf16(w - hi) (w - hi is exact
// in fp32).  The kernels hand each hidden layer on as its logistic r = 1 / (1 + exp(2x))
// instead of tanh(x) = 1 - 2 r, so the layers above it hold W' = -2 W (exact: a sign and
// an exponent) and b' = b + sum_k W[n][k] (summed in fp64 from the given weights and
// rounded once): W' r + b' = W tanh(x) + b.  L2's b' is stored times 2 / ln 2, the scale
// its epilogue applies to the accumulator (one fused multiply-add).
aht_status pack_policy_tc(const MlpDims& m, const TcDims& t, const void* const* W,
                          const void* const* b, int vh, int dtype, uint8_t* dst) {
  if ((dtype == AHT_FP32) != (t.split != 0)) return fail(AHT_EINVAL, "weight dtype differs from the context's population");
  std::fill(dst, dst + t.pol_bytes, (uint8_t)0);
  const int esz = dtype == AHT_FP32 ? 4 : 2;
  const int ins[3] = {m.K, m.H0, m.H1};
  const int outs[3] = {m.H0, m.H1, m.NA + vh};
  std::vector<uint8_t> tmp;
  auto put = [&](uint32_t o_hi, uint32_t o_lo, uint32_t off, float f) {  // a bf16 matrix entry
    const uint16_t hi = bf16_rne(f);
    std::memcpy(dst + o_hi + off, &hi, 2);
    if (t.split) {
      const uint16_t lo = bf16_rne(f - bf16_val(hi));
      std::memcpy(dst + o_lo + off, &lo, 2);
    }
  };
  const double two_over_ln2 = 2.0 / std::log(2.0);
  std::vector<double> rowsum;
  for (int l = 0; l < 3; ++l) {
    const void* src = nullptr;
    if (!W[l] || !b[l]) return fail(AHT_EINVAL, "NULL weight pointer");
    if (!read_host(W[l], (size_t)outs[l] * ins[l] * esz, tmp, &src)) return fail(AHT_ECUDA, "copying weights failed");
    rowsum.assign((size_t)outs[l], 0.0);
    for (int n = 0; n < outs[l]; ++n)
      for (int k = 0; k < ins[l]; ++k) {
        const int64_t i = (int64_t)n * ins[l] + k;
        const float f0 = to_f32(src, i, dtype);
        rowsum[n] += (double)f0;
        const float f = l == 0 ? f0 : -2.0f * f0;  // layers fed by a logistic
        if (l == 0 && !t.sparse) put(t.oW1, t.oW1lo, tc::canon_offset(n, k, t.KP), f);
        if (l == 1) put(t.oW2, t.oW2lo, tc::canon_offset(n, k, m.H0), f);
        if (l == 2) {  // B fragment of chunk k / 16 (see TcDims), remainders for split blocks
          const int kk = k % 16, thr = 4 * n + (kk % 8) / 2;
          const uint32_t off = (uint32_t)(((k / 16) * 32 + thr) * 8 + (kk / 8) * 4 + (kk % 2) * 2);
          put(t.oW3, t.oW3 + (uint32_t)m.H1 * 16u, off, f);
        }
      }
    if (!read_host(b[l], (size_t)outs[l] * esz, tmp, &src)) return fail(AHT_ECUDA, "copying biases failed");
    for (int n = 0; n < outs[l]; ++n) {
      const float f = to_f32(src, n, dtype);
      if (l == 0 && !t.sparse)  // b1: weight of the constant-1 input
        put(t.oW1, t.oW1lo, tc::canon_offset(n, m.K, t.KP), f);
      if (l == 1) {
        const float bk = (float)(((double)f + rowsum[n]) * two_over_ln2);
        std::memcpy(dst + t.ob2 + 4 * n, &bk, 4);
      }
      if (l == 2) {
        const float bf = (float)((double)f + rowsum[n]);
        std::memcpy(dst + t.ob3 + 4 * n, &bf, 4);
      }
    }
  }
  return AHT_OK;
}

// Packs one bf16 policy into its streamed block (dst: w.pol_bytes bytes).  A value row,
// if present, is not used by cross-play and is left out.
aht_status pack_policy_wide(const MlpDims& m, const WideDims& w, const void* const* W,
                            const void* const* b, int vh, uint8_t* dst) {
  std::fill(dst, dst + w.pol_bytes, (uint8_t)0);
  const int ins[3] = {m.K, m.H0, m.H1};
  const int outs[3] = {m.H0, m.H1, m.NA + vh};
  std::vector<uint8_t> tmp;
  auto w1_at = [&](int n, int k) {
    return dst + (size_t)((n / 256) * (w.KP / 16) + k / 16) * kWideChunk + tc::canon_offset(n % 256, k % 16, 16);
  };
  auto w2_at = [&](int n, int k) {
    return dst + (size_t)(w.n_l1 + (n / 256) * (w.H / 16) + k / 16) * kWideChunk +
           tc::canon_offset(n % 256, k % 16, 16);
  };
  for (int l = 0; l < 3; ++l) {
    const void* src = nullptr;
    if (!W[l] || !b[l]) return fail(AHT_EINVAL, "NULL weight pointer");
    if (!read_host(W[l], (size_t)outs[l] * ins[l] * 2, tmp, &src)) return fail(AHT_ECUDA, "copying weights failed");
    const uint16_t* wv = static_cast<const uint16_t*>(src);
    for (int n = 0; n < outs[l]; ++n)
      for (int k = 0; k < ins[l]; ++k) {
        const int64_t i = (int64_t)n * ins[l] + k;
        if (l == 0) std::memcpy(w1_at(n, k), &wv[i], 2);
        if (l == 1) std::memcpy(w2_at(n, k), &wv[i], 2);
        if (l == 2 && n < m.NA) {  // B fragment of chunk k / 16, n-tile n / 8 (see WideDims)
          const float f = to_f32(src, i, AHT_BF16);
          const int kk = k % 16, nt_tiles = (w.NAP + 7) / 8;
          const int t = 4 * (n % 8) + (kk % 8) / 2;                 // thread of the fragment
          const size_t off = ((size_t)((k / 16) * nt_tiles + n / 8) * 32 + t) * 8 + (kk / 8) * 4 + (kk % 2) * 2;
          const uint16_t hb = bf16_rne(f);
          std::memcpy(dst + w.oW3 + off, &hb, 2);
        }
      }
    if (!read_host(b[l], (size_t)outs[l] * 2, tmp, &src)) return fail(AHT_ECUDA, "copying biases failed");
    const uint16_t* bb = static_cast<const uint16_t*>(src);
    for (int n = 0; n < outs[l]; ++n) {
      const float f = to_f32(src, n, AHT_BF16);
      if (l == 0) std::memcpy(w1_at(n, m.K), &bb[n], 2);  // b1: weight of the constant-1 input
      if (l == 1) std::memcpy(dst + w.ob2 + 4 * n, &f, 4);
      if (l == 2 && n < m.NA) std::memcpy(dst + w.ob3 + 4 * n, &f, 4);
    }
  }
  return AHT_OK;
}

// Kernel timer: events around the main kernel of a call (see aht_set_timing).
void timer_fold(aht_ctx* c) {
  for (int i = 0; i < c->n_pending; ++i) {
    float ms = 0.0f;
    if (cudaEventSynchronize(c->ev[2 * i + 1]) == cudaSuccess &&
        cudaEventElapsedTime(&ms, c->ev[2 * i], c->ev[2 * i + 1]) == cudaSuccess) {
      c->timed_ms += ms;
      c->timed_launches += 1;
    }
  }
  c->n_pending = 0;
}

int timer_begin(aht_ctx* c) {
  if (!c->timing) return -1;
  if (c->n_pending == aht_ctx::kTimerPairs) timer_fold(c);
  const int i = c->n_pending++;
  cudaEventRecord(c->ev[2 * i], c->stream);
  return i;
}

void timer_end(aht_ctx* c, int i) {
  if (i >= 0) cudaEventRecord(c->ev[2 * i + 1], c->stream);
}

// The failure-detection hook for the tensor-core call about to launch (it fires once).
void take_expire(aht_ctx* c, int32_t* step, uint64_t* ns) {
  *step = c->dbg_expire_step;
  *ns = c->dbg_expire_ns;
  c->dbg_expire_step = -1;
}

// The test hook's buffer for a call of `steps` steps over `rows` rows: NULL when unset;
// false (and the error set) when it is too small.
bool dbg_buffer(aht_ctx* c, int64_t steps, int64_t rows, float** out) {
  *out = nullptr;
  if (!c->dbg_logits) return true;
  if (steps * rows * 2 * kDbgStride > c->dbg_floats) {
    fail(AHT_EINVAL, "the aht_debug_logits buffer is too small for this call");
    return false;
  }
  *out = c->dbg_logits;
  return true;
}

// Cross-play on the streamed tensor-core kernel: max_steps + 1 launches, one per step
// (the last applies the final transition), then the exact pair means.
aht_status xplay_wide(aht_ctx* c, const int32_t* ego_ids, int32_t n_ego, const int32_t* tm_ids,
                      int32_t n_tm, int32_t P, int32_t max_steps, const aht_xplay_out* out) {
  XpTcArgs a{};
  a.b = batch_of(c);
  a.w = c->wd;
  a.tcw = c->wtcw;
  a.n_ego = n_ego;
  a.n_tm = n_tm;
  a.P = P;
  a.max_steps = max_steps;
  for (int i = 0; i < n_ego; ++i) a.ego_ids[i] = ego_ids[i];
  for (int j = 0; j < n_tm; ++j) a.tm_ids[j] = tm_ids[j];
  a.step0 = (uint32_t)c->step;
  a.n_total = (int64_t)n_ego * n_tm * P;
  a.nsteps = c->xp_nsteps;
  a.returns = out->returns ? out->returns : c->xp_returns;
  a.steps = out->steps;
  a.actions = out->actions;
  if (!dbg_buffer(c, max_steps, a.n_total, &a.dbg_logits)) return AHT_EINVAL;
  const int64_t T0 = ((int64_t)n_tm * P + 127) / 128, T1 = ((int64_t)n_ego * P + 127) / 128;
  take_expire(c, &a.dbg_expire_step, &a.dbg_expire_ns);
  const int64_t tiles0 = n_ego * T0, tiles1 = n_tm * T1;
  // H = 512: two CTAs per tile, each computing one N = 256 block of layers 1 and 2
  a.parts = c->wd.H == 512 ? 2 : 1;
  if ((tiles0 + tiles1) * a.parts > INT32_MAX) return fail(AHT_EINVAL, "too many tiles");
  if (a.parts == 2 && std::max(tiles0, tiles1) * 2 > c->xp_slots)
    return fail(AHT_EINVAL, "more two-part tiles than exchange slots");
  a.xch = c->xp_xch;
  a.xflag = c->xp_xflag;
  const bool turn = c->env.kind == AHT_HANABI || c->env.kind == AHT_MINI_HANABI;
  auto launch = c->env.kind == AHT_HANABI        ? hanabi_xplay_tc
                : c->env.kind == AHT_MINI_HANABI ? minihanabi_xplay_tc
                                                 : overcooked_xplay_tc;
  const int tk = timer_begin(c);
  for (int s = 0; s <= max_steps; ++s) {
    a.s = s;
    a.st_in = c->xp_st[s & 1];
    a.st_out = c->xp_st[(s + 1) & 1];
    a.alive_in = c->xp_alive[s & 1];
    a.alive_out = c->xp_alive[(s + 1) & 1];
    a.act_in = c->xp_act[(s + 1) & 1];
    a.act_out = c->xp_act[s & 1];
    a.zp_in = c->xp_zp[(s + 1) & 1];
    a.zp_out = c->xp_zp[s & 1];
    int64_t grid;
    if (turn) grid = (s & 1) ? tiles1 : tiles0;
    else grid = s < max_steps ? tiles0 + tiles1 : tiles0;
    // a stamp no earlier launch of this context used (0 is the flags' initial value)
    if (++c->xp_stamp >= 0x7FFFFFFFu) c->xp_stamp = 1;
    a.xstamp = c->xp_stamp;
    AHT_CUDA(launch(a, (int)(grid * a.parts), c->wide_smem, c->stream));
  }
  timer_end(c, tk);
  const int64_t n_pairs = (int64_t)n_ego * n_tm;
  if (out->matrix) AHT_CUDA(launch_xp_reduce(a.returns, n_pairs, P, out->matrix, c->stream));
  return AHT_OK;
}

// Cross-play of an LBF context on the tensor-core rollout kernel (tiles of up to 128 envs
// of one pair), then the exact pair means.
aht_status xplay_lbf_tc(aht_ctx* c, const int32_t* ego_ids, int32_t n_ego, const int32_t* tm_ids,
                        int32_t n_tm, int32_t P, int32_t max_steps, float* returns, int32_t* steps,
                        uint8_t* actions, float* matrix) {
  PpoTcArgs ta{};
  ta.b = batch_of(c);
  ta.tc = c->tcd;
  ta.tcw = c->tcw;
  ta.n_envs = c->n_envs;
  ta.step0 = (uint32_t)c->step;
  ta.xp.n_tm = n_tm;
  ta.xp.P = P;
  ta.xp.tpp = (P + 127) / 128;
  ta.xp.max_steps = max_steps;
  ta.xp.n_total = (int64_t)n_ego * n_tm * P;
  for (int i = 0; i < n_ego; ++i) ta.xp.ego_ids[i] = ego_ids[i];
  for (int j = 0; j < n_tm; ++j) ta.xp.tm_ids[j] = tm_ids[j];
  ta.xp.returns = returns;
  ta.xp.steps = steps;
  ta.xp.actions = actions;
  if (!dbg_buffer(c, max_steps, ta.xp.n_total, &ta.dbg_logits)) return AHT_EINVAL;
  const int64_t n_pairs = (int64_t)n_ego * n_tm;
  const int64_t grid = n_pairs * ta.xp.tpp;
  if (grid > INT32_MAX) return fail(AHT_EINVAL, "too many tiles");
  take_expire(c, &ta.dbg_expire_step, &ta.dbg_expire_ns);
  const int tk = timer_begin(c);
  AHT_CUDA(lbf_xplay_tc(ta, (int)grid, c->tc_smem, c->stream));
  timer_end(c, tk);
  if (matrix) AHT_CUDA(launch_xp_reduce(returns, n_pairs, P, matrix, c->stream));
  return AHT_OK;
}

// Tile rows for an M-row launch that fits in shared memory (M multiple of 4).
int fit_rows(const aht_ctx* c, int want) {
  int M = (int)align_up(want, 4);
  while (M > 4 && (size_t)smem_layout(M, c->mlp, c->ops.bytes()).total > c->smem_optin) M = (int)align_up(M / 2, 4);
  return M;
}

// The CUDA-core kernels are latency-bound per CTA: halve the tile (down to 32 rows)
// while every tile of the launch still fits in one wave of resident CTAs, so that more
// SMs, and more CTAs per SM, share the work.  tiles(M): the launch's tile count.
template <class F>
int spread_rows(const aht_ctx* c, int M, int which, F tiles) {
  while (M >= 64) {
    const int M2 = (int)align_up(M / 2, 4);
    const int per_sm = c->ops.occupancy(which, smem_layout(M2, c->mlp, c->ops.bytes()).total);
    if (per_sm < 1 || tiles(M2) > (int64_t)per_sm * c->n_sms) break;
    M = M2;
  }
  return M;
}

}  // namespace

namespace aht {
aht_status set_last_error(aht_status s, const char* msg) { return fail(s, msg); }
}  // namespace aht

extern "C" {

const char* aht_last_error(void) { return g_err.c_str(); }

const char* aht_status_string(aht_status s) {
  switch (s) {
    case AHT_OK: return "ok";
    case AHT_EINVAL: return "invalid argument";
    case AHT_ENOMEM: return "out of device memory";
    case AHT_ECUDA: return "CUDA error";
    case AHT_ETIMEOUT: return "device wait timed out";
    case AHT_EDEVICE: return "device-side error";
  }
  return "unknown status";
}

void aht_destroy(aht_ctx* c) {
  if (!c) return;
  DeviceGuard g(c->device);
  cudaStreamSynchronize(c->stream);
  ctx_free(c->state);
  ctx_free(c->ep_step);
  ctx_free(c->rs_kidx);
  ctx_free(c->rs_hist);
  ctx_free(c->weights);
  ctx_free(c->perm);
  ctx_free(c->tiles);
  ctx_free(c->xp_returns);
  ctx_free(c->last_value);
  ctx_free(c->status);
  if (c->staging) ctx_free_host(c->staging);
  if (c->tc_staging) ctx_free_host(c->tc_staging);
  if (c->wide_staging) ctx_free_host(c->wide_staging);
  ctx_free(c->tcw);
  ctx_free(c->wtcw);
  for (int i = 0; i < 2; ++i) {
    ctx_free(c->xp_st[i]);
    ctx_free(c->xp_act[i]);
    ctx_free(c->xp_zp[i]);
    ctx_free(c->xp_alive[i]);
  }
  ctx_free(c->xp_nsteps);
  ctx_free(c->xp_xch);
  ctx_free(c->xp_xflag);
  if (c->upload_done) cudaEventDestroy(c->upload_done);
  for (auto& e : c->ev)
    if (e) cudaEventDestroy(e);
  delete c;
}

aht_status aht_create(const aht_env_desc* envd, const aht_pop_desc* pop, int64_t n_envs,
                      uint64_t seed, void* cuda_stream, aht_ctx** out) {
  if (!out) return fail(AHT_EINVAL, "out is NULL");
  *out = nullptr;
  DevEnv env;
  aht_status st = check_env(envd, &env);
  if (st != AHT_OK) return st;
  if (!pop || !pop->W || !pop->b) return fail(AHT_EINVAL, "population desc or weight arrays are NULL");
  if (pop->n_policies < 1 || pop->n_policies > 1024) return fail(AHT_EINVAL, "n_policies must be in 1..1024");
  if (pop->obs_dim != env.obs_dim) return fail(AHT_EINVAL, "obs_dim does not match the env (" + std::to_string(env.obs_dim) + ")");
  if (pop->n_actions != env.n_actions) return fail(AHT_EINVAL, "n_actions does not match the env (" + std::to_string(env.n_actions) + ")");
  for (int h : {pop->hidden0, pop->hidden1})
    if (h < 16 || h > 512 || h % 16) return fail(AHT_EINVAL, "hidden sizes must be multiples of 16 in 16..512");
  if (pop->weight_dtype != AHT_FP32 && pop->weight_dtype != AHT_BF16) return fail(AHT_EINVAL, "weight_dtype must be AHT_FP32 or AHT_BF16");
  if (n_envs < 1 || n_envs > (int64_t)1 << 30) return fail(AHT_EINVAL, "n_envs must be in 1..2^30");

  aht_ctx* c = new aht_ctx();
  c->desc = *envd;
  c->env = env;
  c->ops = ops_for(env.kind);
  c->n_policies = pop->n_policies;
  c->n_envs = n_envs;
  c->seed = seed;
  c->step = 0;
  c->stream = (cudaStream_t)cuda_stream;
  c->mlp = make_dims(env.obs_dim, pop->hidden0, pop->hidden1, env.n_actions, env.kind == AHT_LBF);
  auto bail = [&](aht_status s, const std::string& m) {
    aht_destroy(c);
    return fail(s, m);
  };
  if (cudaGetDevice(&c->device) != cudaSuccess) return bail(AHT_ECUDA, "no CUDA device");
  int optin = 0;
  cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, c->device);
  c->smem_optin = (size_t)optin;
  int sms = 0;
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, c->device);
  c->n_sms = sms;

  const MlpDims& m = c->mlp;
  std::vector<float> packed((size_t)m.stride * pop->n_policies, 0.0f);
  for (int p = 0; p < pop->n_policies; ++p) {
    const int vh = pop->has_value_head ? pop->has_value_head[p] : 0;
    aht_status ps = pack_policy(m, pop->W + 3 * p, pop->b + 3 * p, pop->weight_dtype, vh,
                                packed.data() + (size_t)p * m.stride);
    if (ps != AHT_OK) {
      std::string msg = g_err;
      return bail(ps, msg);
    }
  }

  const int words = c->ops.words();
  // the smallest tile any launch uses, plus one partial tile per pool member of the
  // per-episode grouping
  c->max_tiles = group_tiles(n_envs, 4) + kMaxPool;
  struct Alloc { void** p; size_t bytes; };
  Alloc allocs[] = {
      {(void**)&c->state, (size_t)words * n_envs * 4},
      {(void**)&c->ep_step, (size_t)n_envs * 4},
      {(void**)&c->rs_kidx, 2 * (size_t)align_up(n_envs, 16)},
      {(void**)&c->rs_hist, 3 * (size_t)kMaxPool * 4},
      {(void**)&c->weights, packed.size() * 4},
      {(void**)&c->perm, (size_t)n_envs * 4},
      {(void**)&c->tiles, (size_t)c->max_tiles * sizeof(int4)},
      {(void**)&c->xp_returns, (size_t)n_envs * 4},
      {(void**)&c->last_value, (size_t)n_envs * 8},  // V_T scratch of seat 0 and seat 1
      {(void**)&c->status, 4},
  };
  for (auto& a : allocs)
    if (ctx_malloc(a.p, a.bytes) != cudaSuccess) {
      cudaGetLastError();
      return bail(AHT_ENOMEM, "cudaMalloc of " + std::to_string(a.bytes) + " bytes failed");
    }
  if (cudaMemcpy(c->weights, packed.data(), packed.size() * 4, cudaMemcpyHostToDevice) != cudaSuccess ||
      cudaMemset(c->status, 0, 4) != cudaSuccess)
    return bail(AHT_ECUDA, "uploading the population failed");
  if (c->ops.smem_limit(c->smem_optin) != cudaSuccess || policy_set_smem_limit(c->smem_optin) != cudaSuccess)
    return bail(AHT_ECUDA, "setting the shared-memory limit failed");
  if (ctx_malloc_host((void**)&c->staging, (size_t)m.stride * 4) != cudaSuccess)
    return bail(AHT_ENOMEM, "pinned staging allocation failed");
  if (cudaEventCreateWithFlags(&c->upload_done, cudaEventDisableTiming) != cudaSuccess)
    return bail(AHT_ECUDA, "cudaEventCreate failed");
  for (auto& e : c->ev)
    if (cudaEventCreate(&e) != cudaSuccess) return bail(AHT_ECUDA, "cudaEventCreate failed");
  c->weight_dtype = pop->weight_dtype;
  if (tc_eligible(c, pop->weight_dtype)) {
    c->tcd = make_tc_dims(m, pop->weight_dtype == AHT_FP32);
    c->tc_smem = tc_smem_bytes(c->tcd, m.K, c->ops.bytes());
    std::vector<uint8_t> blocks((size_t)c->tcd.pol_bytes * pop->n_policies);
    for (int p = 0; p < pop->n_policies; ++p) {
      const int vh = pop->has_value_head ? pop->has_value_head[p] : 0;
      aht_status ps = pack_policy_tc(m, c->tcd, pop->W + 3 * p, pop->b + 3 * p, vh, pop->weight_dtype,
                                     blocks.data() + (size_t)p * c->tcd.pol_bytes);
      if (ps != AHT_OK) {
        std::string msg = g_err;
        return bail(ps, msg);
      }
    }
    if (ctx_malloc((void**)&c->tcw, blocks.size()) != cudaSuccess) {
      cudaGetLastError();
      return bail(AHT_ENOMEM, "cudaMalloc of the tensor-core population failed");
    }
    if (cudaMemcpy(c->tcw, blocks.data(), blocks.size(), cudaMemcpyHostToDevice) != cudaSuccess)
      return bail(AHT_ECUDA, "uploading the tensor-core population failed");
    if (ctx_malloc_host((void**)&c->tc_staging, c->tcd.pol_bytes) != cudaSuccess)
      return bail(AHT_ENOMEM, "pinned staging allocation failed");
    c->tc = true;
  }
  if (wide_eligible(c, pop->weight_dtype)) {
    c->wd = make_wide_dims(m);
    c->wide_smem = xp_tc_smem_bytes(c->wd);
    std::vector<uint8_t> blocks((size_t)c->wd.pol_bytes * pop->n_policies);
    for (int p = 0; p < pop->n_policies; ++p) {
      const int vh = pop->has_value_head ? pop->has_value_head[p] : 0;
      aht_status ps = pack_policy_wide(m, c->wd, pop->W + 3 * p, pop->b + 3 * p, vh,
                                       blocks.data() + (size_t)p * c->wd.pol_bytes);
      if (ps != AHT_OK) {
        std::string msg = g_err;
        return bail(ps, msg);
      }
    }
    Alloc wa[] = {
        {(void**)&c->wtcw, blocks.size()},
        {(void**)&c->xp_st[0], (size_t)words * n_envs * 4},
        {(void**)&c->xp_st[1], (size_t)words * n_envs * 4},
        {(void**)&c->xp_act[0], (size_t)n_envs * 2},
        {(void**)&c->xp_act[1], (size_t)n_envs * 2},
        {(void**)&c->xp_zp[0], (size_t)n_envs * 2 * 2 * c->wd.NAP * 4},
        {(void**)&c->xp_zp[1], (size_t)n_envs * 2 * 2 * c->wd.NAP * 4},
        {(void**)&c->xp_alive[0], (size_t)n_envs},
        {(void**)&c->xp_alive[1], (size_t)n_envs},
        {(void**)&c->xp_nsteps, (size_t)n_envs * 4},
    };
    for (auto& x : wa)
      if (ctx_malloc(x.p, x.bytes) != cudaSuccess) {
        cudaGetLastError();
        return bail(AHT_ENOMEM, "cudaMalloc of " + std::to_string(x.bytes) + " bytes failed");
      }
    if (cudaMemcpy(c->wtcw, blocks.data(), blocks.size(), cudaMemcpyHostToDevice) != cudaSuccess)
      return bail(AHT_ECUDA, "uploading the streamed tensor-core population failed");
    const cudaError_t se = env.kind == AHT_MINI_HANABI ? minihanabi_xplay_tc_smem_limit(c->wide_smem)
                           : env.kind == AHT_HANABI    ? hanabi_xplay_tc_smem_limit(c->wide_smem)
                                                  : overcooked_xplay_tc_smem_limit(c->wide_smem);
    if (se != cudaSuccess) return bail(AHT_ECUDA, "setting the shared-memory limit failed");
    if (ctx_malloc_host((void**)&c->wide_staging, c->wd.pol_bytes) != cudaSuccess)
      return bail(AHT_ENOMEM, "pinned staging allocation failed");
    if (c->wd.H == 512) {
      // a call's tiles of one seat: at most n_total / 128 + n_ego (or n_tm) <= n_envs / 128 + 64
      c->xp_slots = 2 * ((n_envs + 127) / 128 + kMaxXpIds);
      if (ctx_malloc((void**)&c->xp_xch, (size_t)c->xp_slots * kXchSlot) != cudaSuccess ||
          ctx_malloc((void**)&c->xp_xflag, (size_t)c->xp_slots * 4) != cudaSuccess) {
        cudaGetLastError();
        return bail(AHT_ENOMEM, "cudaMalloc of the cross-play exchange slots failed");
      }
      if (cudaMemset(c->xp_xflag, 0, (size_t)c->xp_slots * 4) != cudaSuccess)
        return bail(AHT_ECUDA, "clearing the cross-play exchange flags failed");
    }
    c->wide = true;
  }
  *out = c;
  aht_status r = aht_reset(c, seed);
  if (r != AHT_OK) {
    *out = nullptr;
    std::string msg = g_err;
    aht_destroy(c);
    return fail(r, msg);
  }
  if (cudaStreamSynchronize(c->stream) != cudaSuccess) {
    *out = nullptr;
    aht_destroy(c);
    return fail(AHT_ECUDA, "reset kernel failed");
  }
  return AHT_OK;
}

aht_status aht_reset(aht_ctx* c, uint64_t seed) {
  if (!c) return fail(AHT_EINVAL, "ctx is NULL");
  DeviceGuard g(c->device);
  c->seed = seed;
  c->step = 0;
  ResetArgs a{batch_of(c), c->state, c->n_envs, 0u, c->ep_step};
  AHT_CUDA(c->ops.reset(a, c->stream));
  return AHT_OK;
}

static aht_status check_traj_out(const aht_traj* out) {
  if (out->advantages && (!out->rewards || !out->values || !out->dones))
    return fail(AHT_EINVAL, "advantages need rewards, values and dones");
  if (out->gamma < 0.f || out->gamma > 1.f || out->lambda < 0.f || out->lambda > 1.f)
    return fail(AHT_EINVAL, "gamma and lambda must be in [0, 1]");
  return AHT_OK;
}

// PPO collection with pool-drawn teammates; out1 (may be NULL) receives seat 1's learner
// trajectory (IPPO).
static aht_status rollout_common(aht_ctx* c, int32_t ego_id, const int32_t* pool, int32_t pool_size,
                                 int32_t T, const aht_traj* out, const aht_traj* out1) {
  if (!c || !out) return fail(AHT_EINVAL, "ctx or out is NULL");
  if (c->env.kind == AHT_HANABI || c->env.kind == AHT_MINI_HANABI)
    return fail(AHT_EINVAL, "PPO collection needs a simultaneous-move env (LBF, Overcooked)");
  if (ego_id < 0 || ego_id >= c->n_policies) return fail(AHT_EINVAL, "ego_id out of range");
  if (!pool || pool_size < 1 || pool_size > kMaxPool) return fail(AHT_EINVAL, "pool_size must be in 1..256");
  for (int k = 0; k < pool_size; ++k) {
    if (pool[k] >= c->n_policies || pool[k] < -AHT_LBF_N_HEURISTICS) return fail(AHT_EINVAL, "pool id out of range");
    if (pool[k] < 0 && !(c->env.kind == AHT_LBF && c->tc))
      return fail(AHT_EINVAL, "heuristic teammates (negative ids) need an LBF context on the tensor-core path");
  }
  if (T < 1) return fail(AHT_EINVAL, "T must be >= 1");
  if (c->step + T + 1 > (int64_t)UINT32_MAX) return fail(AHT_EINVAL, "step counter would exceed 2^32");
  if (aht_status e = check_traj_out(out)) return e;
  if (pool_size > 1 && (reinterpret_cast<uintptr_t>(out->obs) & 3u))
    return fail(AHT_EINVAL, "out->obs must be 4-byte aligned when pool_size > 1");
  if (out1) {
    if (aht_status e = check_traj_out(out1)) return e;
    if (reinterpret_cast<uintptr_t>(out1->obs) & 3u)
      return fail(AHT_EINVAL, "out1->obs must be 4-byte aligned");
  }
  DeviceGuard g(c->device);
  const int64_t Nall = c->n_envs;
  // the sparse-first-layer tensor-core kernel does plain collection; IPPO there runs on
  // the CUDA-core kernel
  const bool use_tc = c->tc && !(c->tcd.sparse && out1);
  // Sec. 3: every env draws its teammate from the pool (once per call); with more than
  // one member the envs are grouped by their draw, so a tile runs one teammate policy
  const bool grouped = pool_size > 1;
  auto n_tiles = [&](int m) -> int64_t {
    return grouped ? resample_tiles(Nall, m, pool_size) : group_tiles(Nall, m);
  };
  int M = 128;
  if (use_tc) {
    // a tensor-core tile's step takes about as long for 32 rows as for 128: while the
    // batch would leave SMs idle, cut the teammate groups into smaller tiles
    while (M > 32 && n_tiles(M / 2) <= c->n_sms) M /= 2;
  } else {
    M = spread_rows(c, fit_rows(c, 128), 0, n_tiles);
  }
  const size_t tc_smem = c->tc_smem + (grouped ? kTcGatherScratch : 0);
  if (use_tc && tc_smem > c->smem_optin) return fail(AHT_EINVAL, "no shared memory left for the teammate grouping");
  float* dbg = nullptr;
  if (use_tc && !dbg_buffer(c, T, Nall, &dbg)) return AHT_EINVAL;
  const int grid = (int)n_tiles(M);

  GroupArgs ga{};
  ga.key = batch_of(c).key;
  ga.n_envs = c->n_envs;
  ga.step0 = (uint32_t)c->step;
  ga.pool_size = pool_size;
  for (int k = 0; k < pool_size; ++k) ga.pool[k] = pool[k];
  ga.M = M;
  ga.max_tiles = grid;
  ga.perm = c->perm;
  ga.tiles = c->tiles;
  ga.teammate = out->teammate;
  if (!grouped) {
    AHT_CUDA(launch_group(ga, c->stream));
  } else if (use_tc) {
    ga.kidx = c->rs_kidx;
    ga.hist = c->rs_hist;
    AHT_CUDA(cudaMemsetAsync(c->rs_hist, 0, (size_t)pool_size * 4, c->stream));
    AHT_CUDA(launch_teammate_draw(ga, c->stream));
  } else {
    ResampleGroupArgs rg{};
    rg.key = ga.key;
    rg.n_envs = Nall;
    rg.step0 = ga.step0;
    rg.ep_step = nullptr;  // per-call draw
    rg.pool_size = pool_size;
    for (int k = 0; k < pool_size; ++k) rg.pool[k] = pool[k];
    rg.M = M;
    rg.max_tiles = grid;
    rg.perm = c->perm;
    rg.tiles = c->tiles;
    rg.teammate = out->teammate;
    AHT_CUDA(launch_resample_group(rg, c->stream));
  }

  PpoArgs a{};
  a.b = batch_of(c);
  a.state = c->state;
  a.n_envs = c->n_envs;
  a.perm = c->perm;
  a.tiles = c->tiles;
  a.M = M;
  a.ego = ego_id;
  a.step0 = (uint32_t)c->step;
  a.T = T;
  a.ep_step = c->ep_step;
  a.traj = TrajPtrs{out->obs, out->actions, out->tm_actions, out->logp, out->values,
                    out->rewards, out->dones,
                    out->last_value ? out->last_value : (out->advantages ? c->last_value : nullptr)};
  if (out1)
    a.traj1 = TrajPtrs{out1->obs, out1->actions, out1->tm_actions, out1->logp, out1->values,
                       out1->rewards, out1->dones,
                       out1->last_value ? out1->last_value
                                        : (out1->advantages ? c->last_value + c->n_envs : nullptr)};
  if (use_tc) {
    PpoTcArgs ta{};
    ta.b = a.b;
    ta.tc = c->tcd;
    ta.tcw = c->tcw;
    ta.state = c->state;
    ta.n_envs = c->n_envs;
    ta.tiles = c->tiles;
    ta.ego = ego_id;
    ta.step0 = a.step0;
    ta.T = T;
    ta.traj = a.traj;
    ta.traj1 = a.traj1;
    ta.ep_step = c->ep_step;
    ta.dbg_logits = dbg;
    take_expire(c, &ta.dbg_expire_step, &ta.dbg_expire_ns);
    if (grouped) {
      ta.gather = 1;
      ta.g.kidx_cur = c->rs_kidx;
      ta.g.hist_cur = c->rs_hist;
      ta.g.scratch_off = (uint32_t)c->tc_smem;
      ta.g.resample = 0;
      ta.g.M = M;
      ta.g.pool_size = pool_size;
      for (int k = 0; k < pool_size; ++k) ta.g.pool[k] = pool[k];
    }
    // a programmatic dependent of the grouping kernel just launched: its CTAs set up and
    // copy the ego's weights while that kernel finishes (the two-group kernel; the others
    // launch in plain stream order)
    ta.pdl = 1;
    const int tk = timer_begin(c);
    AHT_CUDA(lbf_ppo_tc(ta, grid, tc_smem, c->stream));
    timer_end(c, tk);
  } else {
    const size_t smem = smem_layout(M, c->mlp, c->ops.bytes()).total;
    const int tk = timer_begin(c);
    AHT_CUDA(c->ops.ppo(a, grid, smem, c->stream));
    timer_end(c, tk);
  }
  if (out->advantages)
    AHT_CUDA(launch_gae(out->rewards, out->values, out->dones, a.traj.last_value, c->n_envs, T,
                        out->gamma, out->lambda, out->advantages, out->targets, c->stream));
  if (out1 && out1->advantages)
    AHT_CUDA(launch_gae(out1->rewards, out1->values, out1->dones, a.traj1.last_value, c->n_envs, T,
                        out1->gamma, out1->lambda, out1->advantages, out1->targets, c->stream));
  c->step += T;
  return AHT_OK;
}

aht_status aht_rollout(aht_ctx* c, int32_t ego_id, const int32_t* pool, int32_t pool_size,
                       int32_t T, const aht_traj* out) {
  return rollout_common(c, ego_id, pool, pool_size, T, out, nullptr);
}

aht_status aht_rollout_resample(aht_ctx* c, int32_t ego_id, const int32_t* pool, int32_t pool_size,
                                int32_t T, const aht_traj* out, int32_t* teammates) {
  if (!c || !out) return fail(AHT_EINVAL, "ctx or out is NULL");
  if (c->env.kind == AHT_HANABI || c->env.kind == AHT_MINI_HANABI)
    return fail(AHT_EINVAL, "PPO collection needs a simultaneous-move env (LBF, Overcooked)");
  if (ego_id < 0 || ego_id >= c->n_policies) return fail(AHT_EINVAL, "ego_id out of range");
  if (!pool || pool_size < 1 || pool_size > kMaxPool) return fail(AHT_EINVAL, "pool_size must be in 1..256");
  for (int k = 0; k < pool_size; ++k) {
    if (pool[k] >= c->n_policies || pool[k] < -AHT_LBF_N_HEURISTICS) return fail(AHT_EINVAL, "pool id out of range");
    if (pool[k] < 0 && !(c->env.kind == AHT_LBF && c->tc && !c->tcd.sparse))
      return fail(AHT_EINVAL, "heuristic teammates (negative ids) need an LBF context on the tensor-core path "
                              "with the observation in tensor memory");
  }
  if (T < 1) return fail(AHT_EINVAL, "T must be >= 1");
  if (c->step + T + 1 > (int64_t)UINT32_MAX) return fail(AHT_EINVAL, "step counter would exceed 2^32");
  if (aht_status e = check_traj_out(out)) return e;
  if (reinterpret_cast<uintptr_t>(out->obs) & 3u) return fail(AHT_EINVAL, "out->obs must be 4-byte aligned");
  DeviceGuard g(c->device);
  // the gathered per-episode tiles run on the dense-first-layer tensor-core kernel; the
  // sparse-first-layer contexts (LBF beyond 256 tensor-memory columns) on CUDA cores
  const bool use_tc = c->tc && !c->tcd.sparse;
  const int M = use_tc ? 128 : fit_rows(c, 128);
  const int64_t N = c->n_envs;
  const int od = c->env.obs_dim;
  const int grid = resample_tiles(N, M, pool_size);
  float* last_value = out->last_value ? out->last_value : (out->advantages ? c->last_value : nullptr);

  if (use_tc) {
    // Tensor-core path: each step's launch groups its own rows (TcGather).
    const size_t smem = c->tc_smem + kTcGatherScratch;
    if (smem > c->smem_optin) return fail(AHT_EINVAL, "no shared memory left for the per-episode grouping");
    float* dbg = nullptr;
    if (!dbg_buffer(c, T, N, &dbg)) return AHT_EINVAL;
    int32_t expire_step;
    uint64_t expire_ns;
    take_expire(c, &expire_step, &expire_ns);
    const size_t ks = (size_t)align_up(N, 16);
    AHT_CUDA(cudaMemsetAsync(c->rs_hist, 0, 3 * (size_t)kMaxPool * 4, c->stream));
    AHT_CUDA(launch_resample_init(batch_of(c).key, N, c->ep_step, pool_size, c->rs_kidx, c->rs_hist,
                                  c->stream));
    PpoTcArgs ta{};
    ta.b = batch_of(c);
    ta.tc = c->tcd;
    ta.tcw = c->tcw;
    ta.state = c->state;
    ta.n_envs = N;
    ta.ego = ego_id;
    ta.T = 1;
    ta.ep_step = c->ep_step;
    ta.gather = 1;
    ta.g.scratch_off = (uint32_t)c->tc_smem;
    ta.g.resample = 1;
    ta.g.M = 128;
    ta.g.pool_size = pool_size;
    for (int k = 0; k < pool_size; ++k) ta.g.pool[k] = pool[k];
    for (int t = 0; t < T; ++t) {
      const int64_t o = (int64_t)t * N;
      ta.step0 = (uint32_t)(c->step + t);
      ta.traj = TrajPtrs{out->obs ? out->obs + o * od : nullptr, out->actions ? out->actions + o : nullptr,
                         out->tm_actions ? out->tm_actions + o : nullptr, out->logp ? out->logp + o : nullptr,
                         out->values ? out->values + o : nullptr, out->rewards ? out->rewards + o : nullptr,
                         out->dones ? out->dones + o : nullptr, t == T - 1 ? last_value : nullptr};
      ta.g.kidx_cur = c->rs_kidx + (t & 1) * ks;
      ta.g.kidx_next = c->rs_kidx + ((t + 1) & 1) * ks;
      ta.g.hist_cur = c->rs_hist + (t % 3) * kMaxPool;
      ta.g.hist_next = c->rs_hist + ((t + 1) % 3) * kMaxPool;
      ta.g.hist_zero = c->rs_hist + ((t + 2) % 3) * kMaxPool;
      ta.g.teammate = teammates ? teammates + o : nullptr;
      ta.g.teammate2 = t == 0 ? out->teammate : nullptr;
      ta.dbg_logits = dbg ? dbg + o * 2 * kDbgStride : nullptr;  // this step's slice
      ta.dbg_expire_step = t == expire_step ? 0 : -1;             // this launch's step 0
      ta.dbg_expire_ns = expire_ns;
      ta.pdl = t > 0;  // step 0 follows the grouping launch in plain stream order
      const int tk = timer_begin(c);
      AHT_CUDA(lbf_ppo_tc(ta, resample_tiles(N, 128, pool_size), smem, c->stream));
      timer_end(c, tk);
    }
    if (out->advantages)
      AHT_CUDA(launch_gae(out->rewards, out->values, out->dones, last_value, N, T, out->gamma,
                          out->lambda, out->advantages, out->targets, c->stream));
    c->step += T;
    return AHT_OK;
  }

  // CUDA-core path: a grouping launch, then one rollout launch over the groups' tiles.
  ResampleGroupArgs ga{};
  ga.key = batch_of(c).key;
  ga.n_envs = N;
  ga.step0 = (uint32_t)c->step;
  ga.ep_step = c->ep_step;
  ga.pool_size = pool_size;
  for (int k = 0; k < pool_size; ++k) ga.pool[k] = pool[k];
  ga.M = M;
  ga.max_tiles = grid;
  ga.perm = c->perm;
  ga.tiles = c->tiles;
  // One launch per step: group the envs by their episode's teammate, then one step of
  // every group (the envs that finish their episode draw their next teammate from the
  // ep_step the step writes).
  for (int t = 0; t < T; ++t) {
    const int64_t o = (int64_t)t * N;
    ga.teammate = teammates ? teammates + o : nullptr;
    ga.teammate2 = t == 0 ? out->teammate : nullptr;
    AHT_CUDA(launch_resample_group(ga, c->stream));
    TrajPtrs tp{out->obs ? out->obs + o * od : nullptr, out->actions ? out->actions + o : nullptr,
                out->tm_actions ? out->tm_actions + o : nullptr, out->logp ? out->logp + o : nullptr,
                out->values ? out->values + o : nullptr, out->rewards ? out->rewards + o : nullptr,
                out->dones ? out->dones + o : nullptr, t == T - 1 ? last_value : nullptr};
    const uint32_t step = (uint32_t)(c->step + t);
    {
      PpoArgs a{};
      a.b = batch_of(c);
      a.state = c->state;
      a.n_envs = N;
      a.perm = c->perm;
      a.tiles = c->tiles;
      a.M = M;
      a.ego = ego_id;
      a.step0 = step;
      a.T = 1;
      a.ep_step = c->ep_step;
      a.traj = tp;
      const size_t smem = smem_layout(M, c->mlp, c->ops.bytes()).total;
      const int tk = timer_begin(c);
      AHT_CUDA(c->ops.ppo(a, grid, smem, c->stream));
      timer_end(c, tk);
    }
  }
  if (out->advantages)
    AHT_CUDA(launch_gae(out->rewards, out->values, out->dones, last_value, N, T, out->gamma,
                        out->lambda, out->advantages, out->targets, c->stream));
  c->step += T;
  return AHT_OK;
}

aht_status aht_rollout_ippo(aht_ctx* c, int32_t policy0, int32_t policy1, int32_t T,
                            const aht_traj* out0, const aht_traj* out1) {
  if (!c || !out1) return fail(AHT_EINVAL, "ctx or out1 is NULL");
  if (policy1 < 0 || policy1 >= c->n_policies) return fail(AHT_EINVAL, "policy1 out of range");
  return rollout_common(c, policy0, &policy1, 1, T, out0, out1);
}

aht_status aht_xplay_matrix(aht_ctx* c, const int32_t* ego_ids, int32_t n_ego,
                            const int32_t* tm_ids, int32_t n_tm, int32_t envs_per_pair,
                            int32_t max_steps, const aht_xplay_out* out) {
  if (!c || !out) return fail(AHT_EINVAL, "ctx or out is NULL");
  if (!ego_ids || !tm_ids || n_ego < 1 || n_tm < 1 || n_ego > kMaxXpIds || n_tm > kMaxXpIds)
    return fail(AHT_EINVAL, "n_ego and n_tm must be in 1..64");
  for (int i = 0; i < n_ego; ++i)
    if (ego_ids[i] < 0 || ego_ids[i] >= c->n_policies) return fail(AHT_EINVAL, "ego id out of range");
  for (int j = 0; j < n_tm; ++j) {
    if (tm_ids[j] >= c->n_policies || tm_ids[j] < -AHT_LBF_N_HEURISTICS)
      return fail(AHT_EINVAL, "teammate id out of range");
    if (tm_ids[j] < 0 && !(c->env.kind == AHT_LBF && c->tc))
      return fail(AHT_EINVAL, "heuristic teammates (negative ids) need an LBF context on the tensor-core path");
  }
  if (envs_per_pair < 1 || envs_per_pair > (1 << 14)) return fail(AHT_EINVAL, "envs_per_pair must be in 1..16384");
  if (max_steps < 1) return fail(AHT_EINVAL, "max_steps must be >= 1");
  const int64_t n_pairs = (int64_t)n_ego * n_tm;
  const int64_t n_total = n_pairs * envs_per_pair;
  if (n_total > c->n_envs) return fail(AHT_EINVAL, "n_ego*n_tm*envs_per_pair exceeds the context's n_envs");
  if (c->step + max_steps + 1 > (int64_t)UINT32_MAX) return fail(AHT_EINVAL, "step counter would exceed 2^32");
  DeviceGuard g(c->device);
  if (out->actions) AHT_CUDA(cudaMemsetAsync(out->actions, 255, (size_t)max_steps * n_total * 2, c->stream));
  if (c->wide) {
    const aht_status ws = xplay_wide(c, ego_ids, n_ego, tm_ids, n_tm, envs_per_pair, max_steps, out);
    if (ws != AHT_OK) return ws;
    c->step += max_steps;
    return AHT_OK;
  }
  if (c->tc) {  // LBF: the tensor-core rollout kernel in cross-play mode
    const aht_status ts = xplay_lbf_tc(c, ego_ids, n_ego, tm_ids, n_tm, envs_per_pair, max_steps,
                                       out->returns ? out->returns : c->xp_returns, out->steps, out->actions,
                                       out->matrix);
    if (ts != AHT_OK) return ts;
    c->step += max_steps;
    return AHT_OK;
  }
  const int M = spread_rows(c, fit_rows(c, std::min(c->ops.max_rows, envs_per_pair)), 1,
                            [&](int m) { return n_pairs * ((envs_per_pair + m - 1) / m); });
  XpArgs a{};
  a.b = batch_of(c);
  a.n_ego = n_ego;
  a.n_tm = n_tm;
  a.P = envs_per_pair;
  a.max_steps = max_steps;
  for (int i = 0; i < n_ego; ++i) a.ego_ids[i] = ego_ids[i];
  for (int j = 0; j < n_tm; ++j) a.tm_ids[j] = tm_ids[j];
  a.M = M;
  a.tiles_per_pair = (envs_per_pair + M - 1) / M;
  a.step0 = (uint32_t)c->step;
  a.returns = out->returns ? out->returns : c->xp_returns;
  a.steps = out->steps;
  a.actions = out->actions;
  const size_t smem = smem_layout(M, c->mlp, c->ops.bytes()).total;
  const int64_t grid = n_pairs * a.tiles_per_pair;
  if (grid > INT32_MAX) return fail(AHT_EINVAL, "too many tiles");
  const int tk = timer_begin(c);
  AHT_CUDA(c->ops.xplay(a, (int)grid, smem, c->stream));
  timer_end(c, tk);
  if (out->matrix) AHT_CUDA(launch_xp_reduce(a.returns, n_pairs, envs_per_pair, out->matrix, c->stream));
  c->step += max_steps;
  return AHT_OK;
}

}  // extern "C"

// ---- cross-play without context scratch ------------------------------------------------
// The per-env returns that aht_xplay_matrix keeps in context memory sized at aht_create
// live here instead: one file-scope device array that every GPU loading the library
// holds until the process exits.  Host code must not pass the symbol itself to a kernel
// (on the host it names a stand-in, not device memory); it passes the device address
// that cudaGetSymbolAddress returns for the current device, looked up once per device.
namespace {
constexpr int64_t kStaticXpEnvs = AHT_XPLAY_STATIC_MAX_ENVS;
__device__ __align__(256) float g_static_xp_returns[kStaticXpEnvs];
constexpr int kMaxDevices = 64;
std::mutex g_static_mu;
float* g_static_xp_ptr[kMaxDevices] = {};

aht_status static_xp_returns(int device, float** out) {
  if (device < 0 || device >= kMaxDevices) return fail(AHT_EINVAL, "device index above 63");
  std::lock_guard<std::mutex> lock(g_static_mu);
  if (!g_static_xp_ptr[device]) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_static_xp_returns);  // device is current
    if (e != cudaSuccess || !p)
      return fail(AHT_ECUDA, std::string("cudaGetSymbolAddress: ") + cudaGetErrorString(e));
    g_static_xp_ptr[device] = static_cast<float*>(p);
  }
  *out = g_static_xp_ptr[device];
  return AHT_OK;
}
}  // namespace

extern "C" {

aht_status aht_xplay_matrix_static(aht_ctx* c, const int32_t* ego_ids, int32_t n_ego,
                                   const int32_t* tm_ids, int32_t n_tm, int32_t envs_per_pair,
                                   int32_t max_steps, float* matrix) {
  if (!c || !matrix) return fail(AHT_EINVAL, "ctx or matrix is NULL");
  if (!ego_ids || !tm_ids || n_ego < 1 || n_tm < 1 || n_ego > kMaxXpIds || n_tm > kMaxXpIds)
    return fail(AHT_EINVAL, "n_ego and n_tm must be in 1..64");
  for (int i = 0; i < n_ego; ++i)
    if (ego_ids[i] < 0 || ego_ids[i] >= c->n_policies) return fail(AHT_EINVAL, "ego id out of range");
  for (int j = 0; j < n_tm; ++j) {
    if (tm_ids[j] >= c->n_policies || tm_ids[j] < -AHT_LBF_N_HEURISTICS)
      return fail(AHT_EINVAL, "teammate id out of range");
    if (tm_ids[j] < 0 && !(c->env.kind == AHT_LBF && c->tc))
      return fail(AHT_EINVAL, "heuristic teammates (negative ids) need an LBF context on the tensor-core path");
  }
  if (envs_per_pair < 1 || envs_per_pair > (1 << 14)) return fail(AHT_EINVAL, "envs_per_pair must be in 1..16384");
  if (max_steps < 1) return fail(AHT_EINVAL, "max_steps must be >= 1");
  const int64_t n_pairs = (int64_t)n_ego * n_tm;
  const int64_t n_total = n_pairs * envs_per_pair;
  if (n_total > kStaticXpEnvs)
    return fail(AHT_EINVAL, "n_ego*n_tm*envs_per_pair = " + std::to_string(n_total) +
                                " exceeds the static scratch of " + std::to_string(kStaticXpEnvs) + " envs");
  if (c->step + max_steps + 1 > (int64_t)UINT32_MAX) return fail(AHT_EINVAL, "step counter would exceed 2^32");
  DeviceGuard g(c->device);
  float* scratch = nullptr;
  const aht_status ss = static_xp_returns(c->device, &scratch);
  if (ss != AHT_OK) return ss;
  if (c->tc) {  // the same kernel as aht_xplay_matrix, which needs no context scratch here
    const aht_status ts = xplay_lbf_tc(c, ego_ids, n_ego, tm_ids, n_tm, envs_per_pair, max_steps, scratch,
                                       nullptr, nullptr, matrix);
    if (ts != AHT_OK) return ts;
    c->step += max_steps;
    return AHT_OK;
  }
  const int M = spread_rows(c, fit_rows(c, std::min(c->ops.max_rows, envs_per_pair)), 1,
                            [&](int m) { return n_pairs * ((envs_per_pair + m - 1) / m); });
  XpArgs a{};
  a.b = batch_of(c);
  a.n_ego = n_ego;
  a.n_tm = n_tm;
  a.P = envs_per_pair;
  a.max_steps = max_steps;
  for (int i = 0; i < n_ego; ++i) a.ego_ids[i] = ego_ids[i];
  for (int j = 0; j < n_tm; ++j) a.tm_ids[j] = tm_ids[j];
  a.M = M;
  a.tiles_per_pair = (envs_per_pair + M - 1) / M;
  a.step0 = (uint32_t)c->step;
  a.returns = scratch;  // every entry the reduction reads is written first by this call
  a.steps = nullptr;
  a.actions = nullptr;
  const size_t smem = smem_layout(M, c->mlp, c->ops.bytes()).total;
  const int64_t grid = n_pairs * a.tiles_per_pair;
  if (grid > INT32_MAX) return fail(AHT_EINVAL, "too many tiles");
  AHT_CUDA(c->ops.xplay(a, (int)grid, smem, c->stream));
  AHT_CUDA(launch_xp_reduce(scratch, n_pairs, envs_per_pair, matrix, c->stream));
  c->step += max_steps;
  return AHT_OK;
}

aht_status aht_traj_copy(const aht_traj* src, const aht_traj* dst, int64_t n_envs, int32_t T,
                         int32_t obs_dim, void* cuda_stream) {
  if (!src || !dst) return fail(AHT_EINVAL, "src or dst is NULL");
  if (n_envs < 1 || T < 1 || obs_dim < 1) return fail(AHT_EINVAL, "n_envs, T and obs_dim must be >= 1");
  const cudaStream_t st = (cudaStream_t)cuda_stream;
  const size_t steps = (size_t)T * (size_t)n_envs;
  auto copy = [&](void* to, const void* from, size_t bytes) -> bool {
    if (!to || !from) return true;
    return cudaMemcpyAsync(to, from, bytes, cudaMemcpyDefault, st) == cudaSuccess;
  };
  const bool ok = copy(dst->obs, src->obs, steps * (size_t)obs_dim) &&
                  copy(dst->actions, src->actions, steps) && copy(dst->tm_actions, src->tm_actions, steps) &&
                  copy(dst->logp, src->logp, steps * 4) && copy(dst->values, src->values, steps * 4) &&
                  copy(dst->rewards, src->rewards, steps * 4) && copy(dst->dones, src->dones, steps) &&
                  copy(dst->advantages, src->advantages, steps * 4) && copy(dst->targets, src->targets, steps * 4) &&
                  copy(dst->last_value, src->last_value, (size_t)n_envs * 4) &&
                  copy(dst->teammate, src->teammate, (size_t)n_envs * 4);
  if (!ok) {
    const cudaError_t e = cudaGetLastError();
    return fail(AHT_ECUDA, std::string("cudaMemcpyAsync: ") + cudaGetErrorString(e));
  }
  return AHT_OK;
}

aht_status aht_gae(const float* r, const float* v, const uint8_t* d, const float* v_last,
                   int64_t n_envs, int32_t T, float gamma, float lambda, float* adv,
                   float* tgt, void* cuda_stream) {
  if (!r || !v || !d || !v_last || !adv) return fail(AHT_EINVAL, "NULL input or output");
  if (n_envs < 1 || T < 1) return fail(AHT_EINVAL, "n_envs and T must be >= 1");
  if (gamma < 0.f || gamma > 1.f || lambda < 0.f || lambda > 1.f)
    return fail(AHT_EINVAL, "gamma and lambda must be in [0, 1]");
  AHT_CUDA(launch_gae(r, v, d, v_last, n_envs, T, gamma, lambda, adv, tgt, (cudaStream_t)cuda_stream));
  return AHT_OK;
}

aht_status aht_xp_stats(const float* xp, int32_t n_ego, int32_t n_tm, float* upper,
                        const aht_xp_stats_out* out, void* cuda_stream) {
  if (!xp || !upper || !out) return fail(AHT_EINVAL, "NULL matrix, bounds or output struct");
  if (n_ego < 1 || n_tm < 1 || n_ego > AHT_XP_STATS_MAX || n_tm > AHT_XP_STATS_MAX)
    return fail(AHT_EINVAL, "n_ego and n_tm must be in 1..AHT_XP_STATS_MAX");
  if (out->brdiv && n_ego != n_tm) return fail(AHT_EINVAL, "brdiv needs a square matrix");
  static_assert(AHT_XP_STATS_MAX == kXpStatsMax, "cross-play statistics limit");
  XpStatsArgs a{xp, n_ego, n_tm, upper, out->norm, out->regret, out->j_aht, out->j_norm,
                out->max_regret, out->brdiv, out->worst_tm};
  AHT_CUDA(launch_xp_stats(a, (cudaStream_t)cuda_stream));
  return AHT_OK;
}

aht_status aht_debug_tanh(const float* x, float* y, int64_t n, void* cuda_stream) {
  if (!x || !y || n < 1) return fail(AHT_EINVAL, "NULL array or n < 1");
  AHT_CUDA(launch_tanh_probe(x, y, n, (cudaStream_t)cuda_stream));
  return AHT_OK;
}

aht_status aht_step_forced(aht_ctx* c, const uint8_t* actions, const aht_step_out* out) {
  if (!c || !actions || !out) return fail(AHT_EINVAL, "NULL argument");
  if (c->step + 2 > (int64_t)UINT32_MAX) return fail(AHT_EINVAL, "step counter would exceed 2^32");
  DeviceGuard g(c->device);
  ForcedArgs a{batch_of(c), c->state, c->n_envs, (uint32_t)c->step, actions, out->rewards,
               out->team, out->dones, out->obs, c->ep_step};
  AHT_CUDA(c->ops.forced(a, c->stream));
  c->step += 1;
  return AHT_OK;
}

aht_status aht_policy_forward(aht_ctx* c, int32_t policy, const uint8_t* obs, int64_t n,
                              float* out) {
  if (!c || !obs || !out) return fail(AHT_EINVAL, "NULL argument");
  if (policy < 0 || policy >= c->n_policies) return fail(AHT_EINVAL, "policy out of range");
  if (n < 1) return fail(AHT_EINVAL, "n must be >= 1");
  DeviceGuard g(c->device);
  PolicyArgs a{batch_of(c), policy, obs, n, out, 0};
  a.M = fit_rows(c, 64);
  const size_t smem = smem_layout(a.M, c->mlp, 0).total;
  const int64_t grid = (n + a.M - 1) / a.M;
  if (grid > INT32_MAX) return fail(AHT_EINVAL, "n too large");
  AHT_CUDA(launch_policy(a, (int)grid, smem, c->stream));
  return AHT_OK;
}

aht_status aht_get_state(aht_ctx* c, void* buf, size_t* bytes) {
  if (!c || !bytes) return fail(AHT_EINVAL, "NULL argument");
  const size_t body = (size_t)c->ops.words() * c->n_envs * 4, eps = (size_t)c->n_envs * 4;
  const size_t need = sizeof(StateHeader) + body + eps;
  if (!buf) {
    *bytes = need;
    return AHT_OK;
  }
  if (*bytes < need) return fail(AHT_EINVAL, "state buffer too small");
  DeviceGuard g(c->device);
  StateHeader h{kStateMagic, (uint32_t)c->env.kind, (uint32_t)c->ops.words(), 0, c->n_envs, c->seed, c->step};
  std::memcpy(buf, &h, sizeof(h));
  AHT_CUDA(cudaMemcpyAsync(static_cast<uint8_t*>(buf) + sizeof(h), c->state, body, cudaMemcpyDeviceToHost, c->stream));
  AHT_CUDA(cudaMemcpyAsync(static_cast<uint8_t*>(buf) + sizeof(h) + body, c->ep_step, eps,
                           cudaMemcpyDeviceToHost, c->stream));
  AHT_CUDA(cudaStreamSynchronize(c->stream));
  *bytes = need;
  return AHT_OK;
}

aht_status aht_set_state(aht_ctx* c, const void* buf, size_t bytes) {
  if (!c || !buf || bytes < sizeof(StateHeader)) return fail(AHT_EINVAL, "NULL or short buffer");
  StateHeader h;
  std::memcpy(&h, buf, sizeof(h));
  const size_t body = (size_t)c->ops.words() * c->n_envs * 4, eps = (size_t)c->n_envs * 4;
  if (h.magic != kStateMagic || h.kind != (uint32_t)c->env.kind || h.n_words != (uint32_t)c->ops.words() ||
      h.n_envs != c->n_envs || bytes != sizeof(h) + body + eps)
    return fail(AHT_EINVAL, "state buffer does not match this context");
  DeviceGuard g(c->device);
  AHT_CUDA(cudaMemcpyAsync(c->state, static_cast<const uint8_t*>(buf) + sizeof(h), body, cudaMemcpyHostToDevice, c->stream));
  AHT_CUDA(cudaMemcpyAsync(c->ep_step, static_cast<const uint8_t*>(buf) + sizeof(h) + body, eps,
                           cudaMemcpyHostToDevice, c->stream));
  AHT_CUDA(cudaStreamSynchronize(c->stream));
  c->seed = h.seed;
  c->step = h.step;
  return AHT_OK;
}

aht_status aht_set_policy(aht_ctx* c, int32_t policy, const void* const* W, const void* const* b,
                          int32_t weight_dtype, int32_t has_value_head) {
  if (!c || !W || !b) return fail(AHT_EINVAL, "NULL argument");
  if (policy < 0 || policy >= c->n_policies) return fail(AHT_EINVAL, "policy out of range");
  DeviceGuard g(c->device);
  AHT_CUDA(cudaEventSynchronize(c->upload_done));  // the staging buffer is free again
  aht_status ps = pack_policy(c->mlp, W, b, weight_dtype, has_value_head, c->staging);
  if (ps != AHT_OK) return ps;
  AHT_CUDA(cudaMemcpyAsync(c->weights + (int64_t)policy * c->mlp.stride, c->staging,
                           (size_t)c->mlp.stride * 4, cudaMemcpyHostToDevice, c->stream));
  if (c->tc) {
    ps = pack_policy_tc(c->mlp, c->tcd, W, b, has_value_head, weight_dtype, c->tc_staging);
    if (ps != AHT_OK) return ps;
    AHT_CUDA(cudaMemcpyAsync(c->tcw + (int64_t)policy * c->tcd.pol_bytes, c->tc_staging,
                             c->tcd.pol_bytes, cudaMemcpyHostToDevice, c->stream));
  }
  if (c->wide) {
    if (weight_dtype != AHT_BF16) return fail(AHT_EINVAL, "this context's population is bf16");
    ps = pack_policy_wide(c->mlp, c->wd, W, b, has_value_head, c->wide_staging);
    if (ps != AHT_OK) return ps;
    AHT_CUDA(cudaMemcpyAsync(c->wtcw + (int64_t)policy * c->wd.pol_bytes, c->wide_staging,
                             c->wd.pol_bytes, cudaMemcpyHostToDevice, c->stream));
  }
  AHT_CUDA(cudaEventRecord(c->upload_done, c->stream));
  return AHT_OK;
}

aht_status aht_set_timing(aht_ctx* c, int32_t enable) {
  if (!c) return fail(AHT_EINVAL, "ctx is NULL");
  c->timing = enable != 0;
  return AHT_OK;
}

aht_status aht_get_timing(aht_ctx* c, double* kernel_ms, int64_t* launches) {
  if (!c || !kernel_ms || !launches) return fail(AHT_EINVAL, "NULL argument");
  DeviceGuard g(c->device);
  AHT_CUDA(cudaStreamSynchronize(c->stream));
  timer_fold(c);
  *kernel_ms = c->timed_ms;
  *launches = c->timed_launches;
  c->timed_ms = 0.0;
  c->timed_launches = 0;
  return AHT_OK;
}

int64_t aht_step_counter(const aht_ctx* c) { return c ? c->step : -1; }

aht_status aht_sync(aht_ctx* c) {
  if (!c) return fail(AHT_EINVAL, "ctx is NULL");
  DeviceGuard g(c->device);
  AHT_CUDA(cudaStreamSynchronize(c->stream));
  uint32_t s = 0;
  AHT_CUDA(cudaMemcpy(&s, c->status, 4, cudaMemcpyDeviceToHost));
  if (s != 0) {
    AHT_CUDA(cudaMemset(c->status, 0, 4));
    char hex[16];
    std::snprintf(hex, sizeof hex, "%x", s);
    const std::string msg = std::string("device status word 0x") + hex +
                            " (1 illegal action, 2 actor mismatch, 4 bad policy, 8 a bounded wait expired)";
    return fail(s == kStatusTimeout ? AHT_ETIMEOUT : AHT_EDEVICE, msg);
  }
  return AHT_OK;
}

aht_status aht_debug_logits(aht_ctx* c, float* buf, int64_t floats) {
  if (!c) return fail(AHT_EINVAL, "ctx is NULL");
  if (buf && floats < 1) return fail(AHT_EINVAL, "floats must be >= 1");
  c->dbg_logits = buf;
  c->dbg_floats = buf ? floats : 0;
  return AHT_OK;
}

aht_status aht_debug_obs_words(aht_ctx* c, int32_t seat, uint32_t* out) {
  if (!c || !out) return fail(AHT_EINVAL, "ctx or out is NULL");
  if (seat != 0 && seat != 1) return fail(AHT_EINVAL, "seat must be 0 or 1");
  auto launch = c->env.kind == AHT_HANABI        ? hanabi_obs_words
                : c->env.kind == AHT_MINI_HANABI ? minihanabi_obs_words
                : c->env.kind == AHT_OVERCOOKED  ? overcooked_obs_words
                                                 : nullptr;
  if (!launch) return fail(AHT_EINVAL, "LBF observations are not bit rows (LBF cross-play reads bytes)");
  DeviceGuard g(c->device);
  const int words = (c->env.obs_dim + 32) / 32;
  AHT_CUDA(launch(c->state, c->n_envs, batch_of(c).env, seat, words, out, c->stream));
  return AHT_OK;
}

aht_status aht_debug_fail_alloc(int64_t n) {
  g_fail_countdown.store(n > 0 ? n : 0);
  return AHT_OK;
}

int64_t aht_debug_live_allocs(void) { return g_live_allocs.load(); }

aht_status aht_debug_expire_at(aht_ctx* c, int32_t step, int64_t limit_ns) {
  if (!c) return fail(AHT_EINVAL, "ctx is NULL");
  if (step >= 0 && (limit_ns < 1 || limit_ns > 1000000000)) return fail(AHT_EINVAL, "limit_ns must be in 1..1e9");
  c->dbg_expire_step = step < 0 ? -1 : step;
  c->dbg_expire_ns = (uint64_t)limit_ns;
  return AHT_OK;
}

aht_status aht_debug_expire_wait(aht_ctx* c, int64_t limit_ns) {
  if (!c) return fail(AHT_EINVAL, "ctx is NULL");
  if (limit_ns < 1 || limit_ns > 1000000000) return fail(AHT_EINVAL, "limit_ns must be in 1..1e9");
  DeviceGuard g(c->device);
  AHT_CUDA(launch_expire_wait(c->status, (uint64_t)limit_ns, c->stream));
  return AHT_OK;
}

}  // extern "C"

// ======================================================================================
// PPO learner (App. C "PPO ego"): fp32 master weights, Adam moments, the packed bf16 copy
// the gradient kernel loads, per-CTA gradient partials.
// ======================================================================================
struct aht_learner {
  int device = 0;
  cudaStream_t stream = nullptr;
  aht_ppo_config cfg{};
  PpoLayout L{};
  int n_act = 0;
  int max_grid = 0;          // SMs
  int64_t part_stride = 0;   // floats per CTA partial
  int n_blocks = 0;          // reduction blocks
  int64_t t = 0, updates = 0;
  float *params = nullptr, *m = nullptr, *v = nullptr, *partials = nullptr;
  float* mbstat = nullptr;   // [epochs * minibatches][2]
  double *grad = nullptr, *blocksq = nullptr, *advpart = nullptr;
  uint8_t* packed = nullptr;
  uint32_t* status = nullptr;
};

namespace {

PpoLayout ppo_layout(int D, int n_act) {
  PpoLayout L{};
  const int64_t H = kPpoHidden, O = n_act + 1;
  L.D = D;
  L.O = (int32_t)O;
  L.ob1 = H * D;
  L.oW2 = L.ob1 + H;
  L.ob2 = L.oW2 + H * H;
  L.oW3 = L.ob2 + H;
  L.ob3 = L.oW3 + O * H;
  L.n_params = L.ob3 + O;
  return L;
}

void learner_free(aht_learner* L) {
  for (void* p : {(void*)L->params, (void*)L->m, (void*)L->v, (void*)L->partials, (void*)L->mbstat,
                  (void*)L->grad, (void*)L->blocksq, (void*)L->advpart, (void*)L->packed, (void*)L->status})
    if (p) cudaFree(p);
}

aht_status check_traj(const aht_learner* L, const aht_traj* tr, int64_t n_envs, int32_t T) {
  if (!tr || !tr->obs || !tr->actions || !tr->logp || !tr->values || !tr->advantages || !tr->targets)
    return fail(AHT_EINVAL, "traj needs obs, actions, logp, values, advantages and targets");
  if (n_envs < 1 || T < 1) return fail(AHT_EINVAL, "n_envs and T must be >= 1");
  const int64_t S = n_envs * (int64_t)T;
  if (S >= (int64_t(1) << 31)) return fail(AHT_EINVAL, "T * n_envs must be below 2^31");
  if (S % ((int64_t)kPpoTile * L->cfg.minibatches) != 0)
    return fail(AHT_EINVAL, "T * n_envs must be a multiple of 64 * minibatches");
  return AHT_OK;
}

int perm_bits(int64_t S) {
  int w = 2;
  while ((int64_t(1) << w) < S) ++w;
  return w;
}

// One minibatch: grad kernel, reduction, and (step) clip + Adam + repack.
aht_status learner_minibatch(aht_learner* L, const aht_traj* tr, int64_t n_envs, int32_t T,
                             uint32_t epoch, int e, int b, float* stats, bool step) {
  const int64_t S = n_envs * (int64_t)T;
  const uint32_t B = (uint32_t)(S / L->cfg.minibatches);
  const int n_tiles = (int)(B / kPpoTile);
  const int G = std::min(L->max_grid, n_tiles);
  PpoGradArgs a{};
  a.packed = L->packed;
  a.obs = tr->obs;
  a.act = tr->actions;
  a.logp = tr->logp;
  a.val = tr->values;
  a.adv = tr->advantages;
  a.tgt = tr->targets;
  a.D = L->L.D;
  a.n_act = L->n_act;
  a.S = (uint32_t)S;
  a.w = perm_bits(S);
  a.key = Key{(uint32_t)(L->cfg.seed & 0xffffffffu), (uint32_t)(L->cfg.seed >> 32)};
  a.epoch = epoch;
  a.B = B;
  a.mb = (uint32_t)b;
  a.mbstat = L->mbstat + 2 * ((int64_t)e * L->cfg.minibatches + b);
  a.clip_eps = L->cfg.clip_eps;
  a.vf_coef = L->cfg.vf_coef;
  a.ent_coef = L->cfg.ent_coef;
  a.partials = L->partials;
  a.part_stride = L->part_stride;
  a.n_params = L->L.n_params;
  a.oW1 = 0;
  a.ob1 = L->L.ob1;
  a.oW2 = L->L.oW2;
  a.ob2 = L->L.ob2;
  a.oW3 = L->L.oW3;
  a.ob3 = L->L.ob3;
  a.status = L->status;
  AHT_CUDA(launch_ppo_grad(a, G, L->stream));
  PpoAdamArgs ad{};
  ad.L = L->L;
  ad.grad = L->grad;
  ad.blocksq = L->blocksq;
  ad.n_blocks = L->n_blocks;
  ad.params = L->params;
  ad.m = L->m;
  ad.v = L->v;
  ad.packed = L->packed;
  ad.lr = L->cfg.lr;
  ad.b1 = L->cfg.adam_b1;
  ad.b2 = L->cfg.adam_b2;
  ad.eps = L->cfg.adam_eps;
  ad.max_grad_norm = L->cfg.max_grad_norm;
  if (step) {
    L->t += 1;
    ad.c1 = (float)(1.0 - std::pow((double)L->cfg.adam_b1, (double)L->t));
    ad.c2 = (float)(1.0 - std::pow((double)L->cfg.adam_b2, (double)L->t));
  }
  AHT_CUDA(launch_ppo_reduce_adam(L->partials, G, L->part_stride, ad, stats, 1.0f / (float)B, step,
                                  L->stream));
  return AHT_OK;
}

}  // namespace

extern "C" {

aht_status aht_learner_create(int32_t obs_dim, int32_t n_actions, const float* const* W,
                              const float* const* b, const aht_ppo_config* cfg,
                              void* cuda_stream, aht_learner** out) {
  if (!out) return fail(AHT_EINVAL, "out is NULL");
  *out = nullptr;
  if (!W || !b || !cfg) return fail(AHT_EINVAL, "NULL weights or config");
  if (obs_dim < 1 || obs_dim >= kPpoKP || obs_dim % 4 != 0)
    return fail(AHT_EINVAL, "obs_dim must be a multiple of 4 in 4..204");
  if (n_actions < 1 || n_actions + 1 > kPpoMaxOut) return fail(AHT_EINVAL, "n_actions must be in 1..7");
  if (cfg->epochs < 1 || cfg->minibatches < 1) return fail(AHT_EINVAL, "epochs and minibatches must be >= 1");
  if (!(cfg->lr > 0.f) || !(cfg->clip_eps >= 0.f) || !(cfg->adam_eps > 0.f) || !(cfg->adam_b1 >= 0.f) ||
      !(cfg->adam_b1 < 1.f) || !(cfg->adam_b2 >= 0.f) || !(cfg->adam_b2 < 1.f))
    return fail(AHT_EINVAL, "lr, adam_eps > 0; clip_eps >= 0; adam betas in [0, 1)");
  for (int l = 0; l < 3; ++l)
    if (!W[l] || !b[l]) return fail(AHT_EINVAL, "NULL weight pointer");
  auto* L = new aht_learner();
  L->cfg = *cfg;
  L->n_act = n_actions;
  L->L = ppo_layout(obs_dim, n_actions);
  L->stream = (cudaStream_t)cuda_stream;
  auto bail = [&](aht_status st) {
    learner_free(L);
    delete L;
    return st;
  };
  if (cudaGetDevice(&L->device) != cudaSuccess) return bail(fail(AHT_ECUDA, "no CUDA device"));
  cudaDeviceProp prop{};
  if (cudaGetDeviceProperties(&prop, L->device) != cudaSuccess) return bail(fail(AHT_ECUDA, "device query failed"));
  L->max_grid = prop.multiProcessorCount;
  const int64_t np = L->L.n_params;
  L->part_stride = np + 8;
  L->n_blocks = (int)((np + 255) / 256);
  const int n_mb = cfg->epochs * cfg->minibatches;
  bool okm = cudaMalloc(&L->params, np * 4) == cudaSuccess && cudaMalloc(&L->m, np * 4) == cudaSuccess &&
             cudaMalloc(&L->v, np * 4) == cudaSuccess &&
             cudaMalloc(&L->partials, (size_t)L->max_grid * L->part_stride * 4) == cudaSuccess &&
             cudaMalloc(&L->mbstat, (size_t)n_mb * 2 * 4) == cudaSuccess &&
             cudaMalloc(&L->grad, np * 8) == cudaSuccess &&
             cudaMalloc(&L->blocksq, (size_t)L->n_blocks * 8) == cudaSuccess &&
             cudaMalloc(&L->advpart, (size_t)n_mb * kPpoStatBlocks * 2 * 8) == cudaSuccess &&
             cudaMalloc(&L->packed, kPpoPackedBytes) == cudaSuccess && cudaMalloc(&L->status, 4) == cudaSuccess;
  if (!okm) return bail(fail(AHT_ENOMEM, "device allocation failed"));
  const int64_t sizes[6] = {128LL * obs_dim, 128, 128LL * 128, 128, (int64_t)(n_actions + 1) * 128, n_actions + 1};
  const int64_t offs[6] = {0, L->L.ob1, L->L.oW2, L->L.ob2, L->L.oW3, L->L.ob3};
  for (int k = 0; k < 6; ++k) {
    const float* src = (k & 1) ? b[k / 2] : W[k / 2];
    if (cudaMemcpyAsync(L->params + offs[k], src, sizes[k] * 4, cudaMemcpyDefault, L->stream) != cudaSuccess)
      return bail(fail(AHT_ECUDA, "copying the weights failed"));
  }
  if (cudaMemsetAsync(L->m, 0, np * 4, L->stream) != cudaSuccess ||
      cudaMemsetAsync(L->v, 0, np * 4, L->stream) != cudaSuccess ||
      cudaMemsetAsync(L->packed, 0, kPpoPackedBytes, L->stream) != cudaSuccess ||
      cudaMemsetAsync(L->status, 0, 4, L->stream) != cudaSuccess ||
      launch_ppo_pack(L->L, L->params, L->packed, L->stream) != cudaSuccess ||
      ppo_grad_set_smem() != cudaSuccess || cudaStreamSynchronize(L->stream) != cudaSuccess)
    return bail(fail(AHT_ECUDA, "learner initialisation failed"));
  *out = L;
  return AHT_OK;
}

void aht_learner_destroy(aht_learner* L) {
  if (!L) return;
  DeviceGuard g(L->device);
  cudaStreamSynchronize(L->stream);
  learner_free(L);
  delete L;
}

int64_t aht_learner_n_params(const aht_learner* L) { return L ? L->L.n_params : -1; }

aht_status aht_ppo_update(aht_learner* L, const aht_traj* tr, int64_t n_envs, int32_t T, float* stats) {
  if (!L) return fail(AHT_EINVAL, "learner is NULL");
  aht_status st = check_traj(L, tr, n_envs, T);
  if (st != AHT_OK) return st;
  DeviceGuard g(L->device);
  const int64_t S = n_envs * (int64_t)T;
  const int E = L->cfg.epochs, M = L->cfg.minibatches;
  const uint32_t B = (uint32_t)(S / M);
  const uint32_t epoch0 = (uint32_t)(L->updates * E);
  const Key key{(uint32_t)(L->cfg.seed & 0xffffffffu), (uint32_t)(L->cfg.seed >> 32)};
  AHT_CUDA(launch_ppo_advstat(tr->advantages, (uint32_t)S, perm_bits(S), key, epoch0, E, M, B,
                              L->advpart, L->mbstat, L->stream));
  for (int e = 0; e < E; ++e)
    for (int b = 0; b < M; ++b) {
      st = learner_minibatch(L, tr, n_envs, T, epoch0 + (uint32_t)e, e, b,
                             stats ? stats + 6 * ((int64_t)e * M + b) : nullptr, true);
      if (st != AHT_OK) return st;
    }
  L->updates += 1;
  return AHT_OK;
}

aht_status aht_ppo_grad(aht_learner* L, const aht_traj* tr, int64_t n_envs, int32_t T, int32_t epoch,
                        int32_t minibatch, float* grad, float* stats) {
  if (!L || !grad) return fail(AHT_EINVAL, "NULL learner or grad");
  aht_status st = check_traj(L, tr, n_envs, T);
  if (st != AHT_OK) return st;
  if (epoch < 0 || epoch >= L->cfg.epochs || minibatch < 0 || minibatch >= L->cfg.minibatches)
    return fail(AHT_EINVAL, "epoch / minibatch out of range");
  DeviceGuard g(L->device);
  const int64_t S = n_envs * (int64_t)T;
  const int E = L->cfg.epochs, M = L->cfg.minibatches;
  const uint32_t B = (uint32_t)(S / M);
  const uint32_t epoch0 = (uint32_t)(L->updates * E);
  const Key key{(uint32_t)(L->cfg.seed & 0xffffffffu), (uint32_t)(L->cfg.seed >> 32)};
  AHT_CUDA(launch_ppo_advstat(tr->advantages, (uint32_t)S, perm_bits(S), key, epoch0, E, M, B,
                              L->advpart, L->mbstat, L->stream));
  st = learner_minibatch(L, tr, n_envs, T, epoch0 + (uint32_t)epoch, epoch, minibatch, stats, false);
  if (st != AHT_OK) return st;
  AHT_CUDA(launch_f64_to_f32(L->grad, grad, L->L.n_params, L->stream));
  return AHT_OK;
}

aht_status aht_learner_get(aht_learner* L, float* params, float* adam_m, float* adam_v, int64_t* t,
                           int64_t* updates) {
  if (!L) return fail(AHT_EINVAL, "learner is NULL");
  DeviceGuard g(L->device);
  const size_t bytes = (size_t)L->L.n_params * 4;
  if (params) AHT_CUDA(cudaMemcpyAsync(params, L->params, bytes, cudaMemcpyDefault, L->stream));
  if (adam_m) AHT_CUDA(cudaMemcpyAsync(adam_m, L->m, bytes, cudaMemcpyDefault, L->stream));
  if (adam_v) AHT_CUDA(cudaMemcpyAsync(adam_v, L->v, bytes, cudaMemcpyDefault, L->stream));
  if (t) *t = L->t;
  if (updates) *updates = L->updates;
  return AHT_OK;
}

aht_status aht_learner_set(aht_learner* L, const float* params, const float* adam_m, const float* adam_v,
                           int64_t t, int64_t updates) {
  if (!L || !params) return fail(AHT_EINVAL, "NULL learner or params");
  if (t < 0 || updates < 0) return fail(AHT_EINVAL, "t and updates must be >= 0");
  DeviceGuard g(L->device);
  const size_t bytes = (size_t)L->L.n_params * 4;
  AHT_CUDA(cudaMemcpyAsync(L->params, params, bytes, cudaMemcpyDefault, L->stream));
  if (adam_m) AHT_CUDA(cudaMemcpyAsync(L->m, adam_m, bytes, cudaMemcpyDefault, L->stream));
  else AHT_CUDA(cudaMemsetAsync(L->m, 0, bytes, L->stream));
  if (adam_v) AHT_CUDA(cudaMemcpyAsync(L->v, adam_v, bytes, cudaMemcpyDefault, L->stream));
  else AHT_CUDA(cudaMemsetAsync(L->v, 0, bytes, L->stream));
  AHT_CUDA(launch_ppo_pack(L->L, L->params, L->packed, L->stream));
  L->t = t;
  L->updates = updates;
  return AHT_OK;
}

aht_status aht_learner_push(aht_learner* L, aht_ctx* c, int32_t policy) {
  if (!L || !c) return fail(AHT_EINVAL, "NULL learner or ctx");
  DeviceGuard g(L->device);
  AHT_CUDA(cudaStreamSynchronize(L->stream));
  const float* p = L->params;
  if (c->weight_dtype == AHT_FP32) {
    const void* W[3] = {p, p + L->L.oW2, p + L->L.oW3};
    const void* bb[3] = {p + L->L.ob1, p + L->L.ob2, p + L->L.ob3};
    return aht_set_policy(c, policy, W, bb, AHT_FP32, 1);
  }
  // a bf16 population: the nearest-even bf16 of every parameter
  const int64_t n = L->L.n_params;
  std::vector<float> host((size_t)n);
  AHT_CUDA(cudaMemcpy(host.data(), p, (size_t)n * 4, cudaMemcpyDeviceToHost));
  std::vector<uint16_t> h16((size_t)n);
  for (int64_t i = 0; i < n; ++i) h16[(size_t)i] = bf16_rne(host[(size_t)i]);
  const uint16_t* q = h16.data();
  const void* W[3] = {q, q + L->L.oW2, q + L->L.oW3};
  const void* bb[3] = {q + L->L.ob1, q + L->L.ob2, q + L->L.ob3};
  return aht_set_policy(c, policy, W, bb, AHT_BF16, 1);
}

aht_status aht_learner_sync(aht_learner* L) {
  if (!L) return fail(AHT_EINVAL, "learner is NULL");
  DeviceGuard g(L->device);
  AHT_CUDA(cudaStreamSynchronize(L->stream));
  uint32_t s = 0;
  AHT_CUDA(cudaMemcpy(&s, L->status, 4, cudaMemcpyDeviceToHost));
  if (s != 0) {
    AHT_CUDA(cudaMemset(L->status, 0, 4));
    return fail(s == kStatusTimeout ? AHT_ETIMEOUT : AHT_EDEVICE, "learner status word nonzero");
  }
  return AHT_OK;
}

}  // extern "C"
