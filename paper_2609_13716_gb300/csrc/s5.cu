// s5.cu -- one step of the recurrent S5 actor-critic for a batch of envs (the model and
// its readings are stated in include/aht.h).  The dense layers and the SSM's products run
// on this library's tcgen05 GEMM (s5_gemm.cuh) with bf16 operands and fp32 accumulation;
// activations are carried as bf16 terms (hi | lo, or hi | lo | hi against weights
// [Wh | Wh | Wl] for the SSM's fp32 operands) written by each product's epilogue straight
// into the next product's tiled operand, so no fp32 accumulator goes through memory.
#include <cuda_bf16.h>

#include <algorithm>
#include <cmath>
#include <complex>
#include <cstring>
#include <vector>

#include "kernels.h"
#include "s5_gemm.cuh"

namespace aht {
aht_status set_last_error(aht_status s, const char* msg);  // the message of aht_last_error
}  // namespace aht

using namespace aht;

namespace {
// Makes the S5 context's device current for the call (and restores the caller's).
struct S5DeviceGuard {
  int prev = -1;
  explicit S5DeviceGuard(int dev) {
    if (cudaGetDevice(&prev) == cudaSuccess && prev != dev) cudaSetDevice(dev);
    else prev = -1;
  }
  ~S5DeviceGuard() {
    if (prev >= 0) cudaSetDevice(prev);
  }
};
}  // namespace

struct aht_s5 {
  int device = 0;
  cudaStream_t stream = nullptr;
  int K = 0, A = 0, H = 0, P = 0, F = 0;
  int K0 = 0;  // K rounded up to 64: observation columns (and We1 columns) padded with zeros
  int64_t max_n = 0;
  int m_tiles = 0;  // 128-row tiles of max_n
  int n_sms = 0;
  // weights as tiled bf16 GEMM operands (see s5_gemm.cuh).  A layer fed with split
  // activations holds each weight row twice, [W | W] (in = 2I), so that one product over
  // [hi | lo] sums both halves: encoder We1 [H][K0], We2 [H][2H]; SSM Bbar3 [2P][3H]
  // (re rows, then im rows) and Cc3 [H][6P] from Cc = (C_re | -C_im) as [Wh | Wh | Wl];
  // heads Wh0 [2F][2H] (actor rows, then critic), Wh1 and Wh2 [2][F][2F].  The output
  // layers W3a [A][F], W3c [1][F] hold the bf16-rounded weights as fp32.
  uint8_t *We1 = nullptr, *We2 = nullptr, *Bbar3 = nullptr, *Cc3 = nullptr, *Wh0 = nullptr, *Wh1 = nullptr,
          *Wh2 = nullptr;
  float *W3a = nullptr, *W3c = nullptr;
  float *be1 = nullptr, *be2 = nullptr, *bh0 = nullptr, *bh1 = nullptr, *bh2 = nullptr,
        *ba3 = nullptr, *bc3 = nullptr;
  float *lbar = nullptr, *Dv = nullptr;  // lbar [2][P] (re, im), D [H]
  // scratch: tiled activations (x0: the observation; a1..a4: encoder, SSM input and
  // output, residual; a5, a6: [2 heads] of [hi | lo] of F), u fp32 [n][H], head partials
  uint8_t *x0 = nullptr, *a1 = nullptr, *a2 = nullptr, *a3 = nullptr, *a4 = nullptr, *a5 = nullptr,
          *a6 = nullptr;
  float *u = nullptr, *partial = nullptr;
  uint32_t* status = nullptr;
  std::vector<void*> owned;
};

namespace {

#define S5_CUDA(call)                                                                          \
  do {                                                                                         \
    cudaError_t e_ = (call);                                                                   \
    if (e_ != cudaSuccess) return set_last_error(AHT_ECUDA, cudaGetErrorString(e_));          \
  } while (0)

// The observation u8 [n][K] -> the first product's tiled bf16 operand [m_tiles][K0 / 64]
// (exact: small integers), columns K..K0-1 zero; one thread per 8 columns of a row
// (x over a row's chunks, y over rows).
__global__ void obs_tiles(const uint8_t* __restrict__ obs, int K, int K0, int64_t n, uint8_t* __restrict__ x0) {
  const int kc = threadIdx.x;  // 8-column chunk
  if (kc >= K0 / 8) return;
  for (int64_t r = (int64_t)blockIdx.x * blockDim.y + threadIdx.y; r < n; r += (int64_t)gridDim.x * blockDim.y) {
    const uint8_t* row = obs + r * K;
    uint32_t w[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int c = 8 * kc + 2 * j;
      const float f0 = c < K ? (float)row[c] : 0.0f, f1 = c + 1 < K ? (float)row[c + 1] : 0.0f;
      w[j] = tc::pack_bf16(f0, f1);
    }
    const int64_t mt = r >> 7;
    const int rr = (int)(r & 127), kt = kc >> 3, kb = kc & 7;
    *reinterpret_cast<uint4*>(x0 + s5g::chunk_off(mt, K0 / 64, kt, rr, kb)) = make_uint4(w[0], w[1], w[2], w[3]);
  }
}

// logits[e][a] = sum over n-tiles and column halves (in order) of the actor's partial sums
// + ba3[a] (-inf where illegal); values[e] likewise from the critic's
// (slots: the partial sums per (row, head, n-tile, column half): 8, or 32 for A > 8)
__global__ void heads_final(const float* __restrict__ partial, int n_tiles, int slots, const float* __restrict__ ba3,
                            const float* __restrict__ bc3, const uint8_t* __restrict__ legal, int A, int64_t n,
                            float* __restrict__ logits, float* __restrict__ values) {
  const int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (e >= n) return;
  const int parts = 2 * n_tiles;  // (n-tile, column half) pairs
  const float* pa = partial + (e * 2 + 0) * (int64_t)parts * slots;
  const float* pc = partial + (e * 2 + 1) * (int64_t)parts * slots;
  for (int a = 0; a < A; ++a) {
    float z = 0.0f;
    for (int t = 0; t < parts; ++t) z += pa[t * slots + a];
    z += ba3[a];
    logits[e * A + a] = (legal && !legal[e * A + a]) ? -INFINITY : z;
  }
  float v = 0.0f;
  for (int t = 0; t < parts; ++t) v += pc[t * slots];
  values[e] = v + bc3[0];
}

// Output columns per GEMM tile for an N-column product: the widest multiple of 32 up to
// 256 that divides N (N is a multiple of 32).
int bn_for(int N) {
  for (int b = 256; b >= 32; b -= 32)
    if (N % b == 0) return b;
  return 32;
}

// Tiles of a bf16 matrix [rows][cols] (row-major, cols padded with zeros to a multiple of
// 64) for the GEMM: n-tiles of BN rows (rows a multiple of BN), k-tiles of 64.
std::vector<__nv_bfloat16> tile_matrix(const std::vector<__nv_bfloat16>& w, int rows, int cols, int BN) {
  const int KT = (cols + 63) / 64, NT = rows / BN;
  std::vector<__nv_bfloat16> t((size_t)NT * KT * BN * 64, __float2bfloat16_rn(0.0f));
  for (int r = 0; r < rows; ++r)
    for (int c = 0; c < cols; ++c) {
      const int nt = r / BN, rr = r % BN, kt = c / 64, kk = c % 64;
      const size_t tile = ((size_t)nt * KT + kt) * BN * 64;
      const size_t off = (size_t)((rr >> 3) * 8 + (kk >> 3)) * 64 + (rr & 7) * 8 + (kk & 7);
      t[tile + off] = w[(size_t)r * cols + c];
    }
  return t;
}

aht_status run_gemm(aht_s5* s, const s5g::GemmArgs& g0, int64_t n) {
  s5g::GemmArgs g = g0;
  g.n = n;
  g.m_tiles = (int)((n + s5g::kBM - 1) / s5g::kBM);
  g.status = s->status;
  const int tiles = g.m_tiles * g.n_tiles * g.batch;
  const int grid = std::min(tiles, s->n_sms);
  const size_t smem = s5g::gemm_smem_bytes(g.BN);
  if (g.epi == s5g::kHeads && (g.n_out[0] > 8 || g.n_out[1] > 8))
    s5g::gemm_kernel<s5g::kMaxOut><<<grid, s5g::kThreads, smem, s->stream>>>(g);
  else
    s5g::gemm_kernel<8><<<grid, s5g::kThreads, smem, s->stream>>>(g);
  S5_CUDA(cudaGetLastError());
  return AHT_OK;
}

}  // namespace

extern "C" {

aht_status aht_s5_create(const aht_s5_params* p, int64_t max_envs, void* cuda_stream, aht_s5** out) {
  if (!out) return set_last_error(AHT_EINVAL, "out is NULL");
  *out = nullptr;
  if (!p) return set_last_error(AHT_EINVAL, "params is NULL");
  if (p->obs_dim < 1 || p->obs_dim > 2048 || p->n_actions < 1 || p->n_actions > 32 || p->H < 32 ||
      p->H % 32 || p->P < 32 || p->P % 32 || p->P > 128 || p->F < 32 || p->F % 32)
    return set_last_error(AHT_EINVAL,
                          "S5 sizes: 1 <= obs_dim <= 2048, 1 <= n_actions <= 32, H, P, F multiples of 32, P <= 128");
  if (max_envs < 1 || max_envs > (1 << 20)) return set_last_error(AHT_EINVAL, "max_envs must be in 1..2^20");
  const float* req[] = {p->We1, p->be1, p->We2, p->be2, p->lam_re, p->lam_im, p->log_dt, p->B_re,
                        p->B_im, p->C_re, p->C_im, p->D};
  for (const float* q : req)
    if (!q) return set_last_error(AHT_EINVAL, "NULL parameter array");
  for (int l = 0; l < 4; ++l)
    if (!p->Wa[l] || !p->ba[l] || !p->Wc[l] || !p->bc[l]) return set_last_error(AHT_EINVAL, "NULL head array");
  for (int q = 0; q < p->P; ++q)
    if (!(p->lam_re[q] < 0.0f)) return set_last_error(AHT_EINVAL, "lam_re must be negative");

  aht_s5* s = new aht_s5();
  const int K = p->obs_dim, A = p->n_actions, H = p->H, P = p->P, F = p->F;
  s->K = K; s->A = A; s->H = H; s->P = P; s->F = F;
  s->K0 = (K + 63) / 64 * 64;
  s->max_n = max_envs;
  s->m_tiles = (int)((max_envs + s5g::kBM - 1) / s5g::kBM);
  s->stream = static_cast<cudaStream_t>(cuda_stream);
  cudaGetDevice(&s->device);
  cudaDeviceGetAttribute(&s->n_sms, cudaDevAttrMultiProcessorCount, s->device);
  auto bail = [&](aht_status st, const char* msg) {
    aht_s5_destroy(s);
    return set_last_error(st, msg);
  };
  auto alloc = [&](void** ptr, size_t bytes) {
    if (cudaMalloc(ptr, bytes) != cudaSuccess) {
      cudaGetLastError();
      return false;
    }
    s->owned.push_back(*ptr);
    return true;
  };
  auto up = [&](void** dst, const void* h, size_t bytes) {
    return alloc(dst, bytes) && cudaMemcpy(*dst, h, bytes, cudaMemcpyHostToDevice) == cudaSuccess;
  };
  auto bf = [](float x) { return __float2bfloat16_rn(x); };
  // a tiled GEMM operand from an fp32 matrix [rows][cols] given by parts of columns:
  // each part (pointer, its column count, 0: as is, 1: its bf16 remainder w - bf16(w))
  struct Part { const float* w; int cols; int lo; };
  auto tiles_of = [&](int rows, const std::vector<Part>& parts, int row_stride_of_parts) {
    int cols = 0;
    for (const Part& q : parts) cols += q.cols;
    std::vector<__nv_bfloat16> m((size_t)rows * cols);
    for (int r = 0; r < rows; ++r) {
      int c0 = 0;
      for (const Part& q : parts) {
        for (int c = 0; c < q.cols; ++c) {
          const float x = q.w[(size_t)r * row_stride_of_parts + c];
          const __nv_bfloat16 hi = bf(x);
          m[(size_t)r * cols + c0 + c] = q.lo ? bf(x - __bfloat162float(hi)) : hi;
        }
        c0 += q.cols;
      }
    }
    return tile_matrix(m, rows, cols, bn_for(rows));
  };
  auto up_tiled = [&](uint8_t** dst, int rows, const std::vector<Part>& parts, int row_stride_of_parts) {
    const std::vector<__nv_bfloat16> t = tiles_of(rows, parts, row_stride_of_parts);
    return up((void**)dst, t.data(), t.size() * 2);
  };
  auto vec = [](const float* a, size_t n) { return std::vector<float>(a, a + n); };
  auto bf16_rounded = [](const float* a, size_t n) {
    std::vector<float> v(n);
    for (size_t i = 0; i < n; ++i) v[i] = __bfloat162float(__float2bfloat16_rn(a[i]));
    return v;
  };
  auto cat = [](std::vector<float> a, const std::vector<float>& b) {
    a.insert(a.end(), b.begin(), b.end());
    return a;
  };
  auto up32 = [&](float** dst, const std::vector<float>& h) { return up((void**)dst, h.data(), h.size() * 4); };
  // heads: actor rows, then critic rows, of one layer [F][I] as one matrix [2F][I]
  auto stack = [](const float* a, const float* c, size_t n) {
    std::vector<float> v(a, a + n);
    v.insert(v.end(), c, c + n);
    return v;
  };
  const std::vector<float> h0 = stack(p->Wa[0], p->Wc[0], (size_t)F * H);
  bool ok = up_tiled(&s->We1, H, {{p->We1, K, 0}}, K) &&
            up_tiled(&s->We2, H, {{p->We2, H, 0}, {p->We2, H, 0}}, H) &&
            up_tiled(&s->Wh0, 2 * F, {{h0.data(), H, 0}, {h0.data(), H, 0}}, H);
  // the two heads' layers 1 and 2, each a two-member batch: actor tiles, then critic's
  for (int l = 1; ok && l <= 2; ++l) {
    std::vector<__nv_bfloat16> both;
    for (int h = 0; h < 2; ++h) {
      const float* w = h ? p->Wc[l] : p->Wa[l];
      const std::vector<__nv_bfloat16> t = tiles_of(F, {{w, F, 0}, {w, F, 0}}, F);
      both.insert(both.end(), t.begin(), t.end());
    }
    ok = up((void**)(l == 1 ? &s->Wh1 : &s->Wh2), both.data(), both.size() * 2);
  }
  if (!ok) return bail(AHT_ENOMEM, "S5 weight upload failed");
  ok = up32(&s->W3a, bf16_rounded(p->Wa[3], (size_t)A * F)) && up32(&s->W3c, bf16_rounded(p->Wc[3], F)) &&
       up32(&s->be1, vec(p->be1, H)) && up32(&s->be2, vec(p->be2, H)) &&
       up32(&s->bh0, cat(vec(p->ba[0], F), vec(p->bc[0], F))) &&
       up32(&s->bh1, cat(vec(p->ba[1], F), vec(p->bc[1], F))) &&
       up32(&s->bh2, cat(vec(p->ba[2], F), vec(p->bc[2], F))) && up32(&s->ba3, vec(p->ba[3], A)) &&
       up32(&s->bc3, vec(p->bc[3], 1)) && up32(&s->Dv, vec(p->D, H));
  if (!ok) return bail(AHT_ENOMEM, "S5 weight upload failed");
  // zero-order hold in fp64
  std::vector<float> lbar(2 * P), Bbar((size_t)2 * P * H), Cc((size_t)H * 2 * P);
  for (int q = 0; q < P; ++q) {
    const std::complex<double> lam(p->lam_re[q], p->lam_im[q]);
    const std::complex<double> lb = std::exp(lam * std::exp((double)p->log_dt[q]));
    const std::complex<double> sc = (lb - 1.0) / lam;
    lbar[q] = (float)lb.real();
    lbar[P + q] = (float)lb.imag();
    for (int h = 0; h < H; ++h) {
      const std::complex<double> b = sc * std::complex<double>(p->B_re[(size_t)q * H + h], p->B_im[(size_t)q * H + h]);
      Bbar[(size_t)q * H + h] = (float)b.real();
      Bbar[(size_t)(P + q) * H + h] = (float)b.imag();
    }
  }
  for (int h = 0; h < H; ++h)
    for (int q = 0; q < P; ++q) {
      Cc[(size_t)h * 2 * P + q] = p->C_re[(size_t)h * P + q];
      Cc[(size_t)h * 2 * P + P + q] = -p->C_im[(size_t)h * P + q];
    }
  // three-term rows [Wh | Wh | Wl] of the SSM's fp32 matrices
  if (!up32(&s->lbar, lbar) ||
      !up_tiled(&s->Bbar3, 2 * P, {{Bbar.data(), H, 0}, {Bbar.data(), H, 0}, {Bbar.data(), H, 1}}, H) ||
      !up_tiled(&s->Cc3, H, {{Cc.data(), 2 * P, 0}, {Cc.data(), 2 * P, 0}, {Cc.data(), 2 * P, 1}}, 2 * P))
    return bail(AHT_ENOMEM, "S5 upload failed");
  // scratch: tiled activations, zeroed once (their padding columns are never written)
  const int64_t rows = (int64_t)s->m_tiles * s5g::kBM;
  auto kp = [](int k) { return (size_t)((k + 63) / 64 * 64); };
  struct Act { uint8_t** p; size_t bytes; };
  const Act acts[] = {{&s->x0, rows * kp(K) * 2},      {&s->a1, rows * kp(2 * H) * 2},
                      {&s->a2, rows * kp(3 * H) * 2},  {&s->a3, rows * kp(6 * P) * 2},
                      {&s->a4, rows * kp(2 * H) * 2},  {&s->a5, 2 * rows * kp(2 * F) * 2},
                      {&s->a6, 2 * rows * kp(2 * F) * 2}};
  for (const Act& x : acts)
    if (!alloc((void**)x.p, x.bytes) || cudaMemset(*x.p, 0, x.bytes) != cudaSuccess)
      return bail(AHT_ENOMEM, "S5 scratch allocation failed");
  const int n_tiles_f = F / bn_for(F);
  if (!alloc((void**)&s->u, (size_t)rows * H * 4) ||
      !alloc((void**)&s->partial, (size_t)rows * 2 * n_tiles_f * 2 * s5g::kMaxOut * 4) ||
      !alloc((void**)&s->status, 4) || cudaMemset(s->status, 0, 4) != cudaSuccess)
    return bail(AHT_ENOMEM, "S5 scratch allocation failed");
  if (cudaFuncSetAttribute(s5g::gemm_kernel<8>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)s5g::gemm_smem_bytes(256)) != cudaSuccess ||
      cudaFuncSetAttribute(s5g::gemm_kernel<s5g::kMaxOut>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)s5g::gemm_smem_bytes(256)) != cudaSuccess)
    return bail(AHT_ECUDA, "setting the GEMM's shared-memory limit failed");
  *out = s;
  return AHT_OK;
}

void aht_s5_destroy(aht_s5* s) {
  if (!s) return;
  S5DeviceGuard g(s->device);
  for (void* q : s->owned) cudaFree(q);
  delete s;
}

aht_status aht_s5_step(aht_s5* s, const uint8_t* obs, const uint8_t* reset, const uint8_t* legal,
                       int64_t n, float* state, float* logits, float* values) {
  if (!s || !obs || !reset || !state || !logits || !values) return set_last_error(AHT_EINVAL, "NULL argument");
  if (n < 1 || n > s->max_n) return set_last_error(AHT_EINVAL, "n must be in 1..max_envs");
  S5DeviceGuard dg(s->device);
  const int K = s->K, A = s->A, H = s->H, P = s->P, F = s->F;
  const int64_t rows = (int64_t)s->m_tiles * s5g::kBM;
  auto kt = [](int k) { return (k + 63) / 64; };
  // the observation -> tiled bf16
  {
    const int bx = s->K0 / 8, by = std::max(1, 256 / bx);  // K0 <= 2048 keeps bx <= 256
    const int64_t blocks = std::min<int64_t>((n + by - 1) / by, 65535);
    obs_tiles<<<(unsigned)blocks, dim3((unsigned)bx, (unsigned)by), 0, s->stream>>>(obs, K, s->K0, n, s->x0);
    S5_CUDA(cudaGetLastError());
  }
  auto layer = [&](const uint8_t* A_, int k_in, const uint8_t* B_, int N, int epi) {
    s5g::GemmArgs g{};
    g.A = A_;
    g.B = B_;
    g.k_tiles = kt(k_in);
    g.BN = bn_for(N);
    g.n_tiles = N / g.BN;
    g.batch = 1;
    g.epi = epi;
    return g;
  };
  // encoder layer 1 (exact bf16 observation): relu, hi | lo
  s5g::GemmArgs g = layer(s->x0, K, s->We1, H, s5g::kSplit);
  g.bias = s->be1; g.relu = 1; g.parts = 2; g.I = H; g.out = s->a1; g.out_k_tiles = kt(2 * H);
  if (aht_status e = run_gemm(s, g, n)) return e;
  // encoder layer 2: relu; u (fp32) and its hi | lo | hi for the three-term SSM product
  g = layer(s->a1, 2 * H, s->We2, H, s5g::kSplit);
  g.bias = s->be2; g.relu = 1; g.parts = 3; g.I = H; g.out = s->a2; g.out_k_tiles = kt(3 * H); g.out32 = s->u;
  if (aht_status e = run_gemm(s, g, n)) return e;
  // SSM: Bbar u, the recurrence and x's hi | lo | hi
  g = layer(s->a2, 3 * H, s->Bbar3, 2 * P, s5g::kSsm);
  g.lbar = s->lbar; g.state = state; g.reset = reset; g.P = P; g.out = s->a3; g.out_k_tiles = kt(6 * P);
  if (aht_status e = run_gemm(s, g, n)) return e;
  // Re(C x), then v = u + gelu(y + D u) as hi | lo
  g = layer(s->a3, 6 * P, s->Cc3, H, s5g::kGelu);
  g.u = s->u; g.D = s->Dv; g.I = H; g.out = s->a4; g.out_k_tiles = kt(2 * H);
  if (aht_status e = run_gemm(s, g, n)) return e;
  // heads layer 0, both heads at once: relu, hi | lo of each head's F units
  const int64_t head_act = rows * kt(2 * F) * 64 * 2;  // bytes of one head's activation
  g = layer(s->a4, 2 * H, s->Wh0, 2 * F, s5g::kSplit);
  g.bias = s->bh0; g.relu = 1; g.parts = 2; g.I = F; g.out = s->a5; g.out_stride = head_act;
  g.out_k_tiles = kt(2 * F);
  if (aht_status e = run_gemm(s, g, n)) return e;
  // heads layer 1 (two-member batch)
  const int64_t wh_bytes = (int64_t)F * 2 * F * 2;
  g = layer(s->a5, 2 * F, s->Wh1, F, s5g::kSplit);
  g.batch = 2; g.a_stride = head_act; g.b_stride = wh_bytes;
  g.bias = s->bh1; g.relu = 1; g.parts = 2; g.I = F; g.out = s->a6; g.out_stride = head_act;
  g.out_k_tiles = kt(2 * F);
  if (aht_status e = run_gemm(s, g, n)) return e;
  // heads layer 2 with both output layers: per-tile partial sums
  g = layer(s->a6, 2 * F, s->Wh2, F, s5g::kHeads);
  g.batch = 2; g.a_stride = head_act; g.b_stride = wh_bytes;
  g.bias = s->bh2; g.W3[0] = s->W3a; g.W3[1] = s->W3c; g.n_out[0] = A; g.n_out[1] = 1; g.partial = s->partial;
  if (aht_status e = run_gemm(s, g, n)) return e;
  heads_final<<<(unsigned)((n + 255) / 256), 256, 0, s->stream>>>(s->partial, F / bn_for(F), A > 8 ? s5g::kMaxOut : 8,
                                                                  s->ba3, s->bc3, legal, A, n, logits, values);
  S5_CUDA(cudaGetLastError());
  return AHT_OK;
}

aht_status aht_s5_sync(aht_s5* s) {
  if (!s) return set_last_error(AHT_EINVAL, "NULL argument");
  S5DeviceGuard g(s->device);
  S5_CUDA(cudaStreamSynchronize(s->stream));
  uint32_t st = 0;
  S5_CUDA(cudaMemcpy(&st, s->status, 4, cudaMemcpyDeviceToHost));
  if (st) {
    cudaMemset(s->status, 0, 4);
    return set_last_error(AHT_ETIMEOUT, "an S5 GEMM's bounded wait expired");
  }
  return AHT_OK;
}

}  // extern "C"
