// s5.cu -- one step of the recurrent S5 actor-critic for a batch of envs (the model and
// its readings are stated in include/aht.h).  The dense layers are plain GEMMs over the
// batch (cuBLAS, bf16 operands, fp32 accumulate) with the activations carried as two bf16
// halves; the elementwise parts (bias, relu, the split, the SSM recurrence, GELU, masking)
// are this file's kernels.
#include <cublas_v2.h>
#include <cuda_bf16.h>

#include <algorithm>
#include <cmath>
#include <complex>
#include <cstring>
#include <vector>

#include "kernels.h"

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
  cublasHandle_t blas = nullptr;
  int K = 0, A = 0, H = 0, P = 0, F = 0;
  int Kp = 0;  // K rounded up to 16: observation rows and We1 rows padded with zeros
  int64_t max_n = 0;
  // bf16 weights [out][in]. A layer fed with split activations holds each weight row twice,
  // [W | W] (in = 2I), so that one product over [hi | lo] sums both halves. Heads: layer 0
  // [2F][2H] (actor rows, then critic), layers 1-2 [2][F][2F]; the encoder's layer 1 [H][K]
  // sees exact bf16 observations. The output layers, W3 [A + 1][F] (actor rows, then the
  // critic's), hold the bf16-rounded weights as fp32 for the CUDA-core output kernel.
  __nv_bfloat16 *We1 = nullptr, *We2 = nullptr, *Wh0 = nullptr, *Wh1 = nullptr, *Wh2 = nullptr;
  float* W3 = nullptr;
  float *be1 = nullptr, *be2 = nullptr, *bh0 = nullptr, *bh1 = nullptr, *bh2 = nullptr,
        *ba3 = nullptr, *bc3 = nullptr;
  // SSM: lbar [2][P] (re, im) and D [H] fp32.  Its products run as three bf16 terms: an
  // fp32 operand a = ah + al (two bf16), activations stored [hi | lo | hi] and weights
  // [Wh | Wh | Wl], one GEMM sums Wh hi + Wh lo + Wl hi (~2^-16 relative).  Bbar3 [2P][3H]
  // (re rows, then im rows), Cc3 [H][3 x 2P] from Cc = (C_re | -C_im).
  float *lbar = nullptr, *Dv = nullptr;
  __nv_bfloat16 *Bbar3 = nullptr, *Cc3 = nullptr;
  // scratch
  // x16 [n][Kp]; act: split activations, each row [group][hi | lo][I] (heads: 2 groups of F)
  __nv_bfloat16 *x16 = nullptr, *act = nullptr;
  float *acc = nullptr, *u = nullptr, *bu = nullptr, *y = nullptr;
  void* workspace = nullptr;
  std::vector<void*> owned;
};

namespace {

#define S5_CUDA(call)                                                                          \
  do {                                                                                         \
    cudaError_t e_ = (call);                                                                   \
    if (e_ != cudaSuccess) return set_last_error(AHT_ECUDA, cudaGetErrorString(e_));          \
  } while (0)
#define S5_BLAS(call)                                                                          \
  do {                                                                                         \
    if ((call) != CUBLAS_STATUS_SUCCESS) return set_last_error(AHT_ECUDA, "cuBLAS call failed"); \
  } while (0)

constexpr size_t kWorkspace = 32u << 20;

// out[r][c] = obs[r][c] as bf16 for c < K, 0 for K <= c < Kp (Kp % 4 == 0); four columns
// a thread
__global__ void u8_to_bf16(const uint8_t* __restrict__ in, __nv_bfloat16* __restrict__ out, int K, int Kp,
                           int64_t n) {
  const int c = 4 * (blockIdx.x * blockDim.x + threadIdx.x);
  if (c >= Kp) return;
  for (int64_t r = (int64_t)blockIdx.y * blockDim.y + threadIdx.y; r < n; r += (int64_t)gridDim.y * blockDim.y) {
    const uint8_t* row = in + r * K;
    float v[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) v[k] = c + k < K ? (float)row[c + k] : 0.0f;
    __nv_bfloat162 a = __floats2bfloat162_rn(v[0], v[1]), b = __floats2bfloat162_rn(v[2], v[3]);
    *reinterpret_cast<uint2*>(out + r * Kp + c) =
        make_uint2(*reinterpret_cast<uint32_t*>(&a), *reinterpret_cast<uint32_t*>(&b));
  }
}

// Row-wise kernels run on 2-D blocks and grids: x covers a row's columns (four per thread;
// the widths are multiples of 16), y strides over rows, so that column arithmetic stays
// 32-bit.
constexpr int kRowsPerThread = 4;  // rows a thread of bias_act_split loads before it stores

__device__ __forceinline__ int64_t row0() { return (int64_t)blockIdx.y * blockDim.y + threadIdx.y; }
__device__ __forceinline__ int64_t row_step() { return (int64_t)gridDim.y * blockDim.y; }

__device__ __forceinline__ uint2 pack_bf16x4(float a, float b, float c, float d) {
  __nv_bfloat162 lo = __floats2bfloat162_rn(a, b), hi = __floats2bfloat162_rn(c, d);
  return make_uint2(*reinterpret_cast<uint32_t*>(&lo), *reinterpret_cast<uint32_t*>(&hi));
}

// writes v (four columns) as hi at d and lo = bf16(v - hi) at d + I (and hi again at
// d + 2I for a three-term product)
__device__ __forceinline__ void store_split4(__nv_bfloat16* d, int I, float4 v, bool hi_again = false) {
  const uint2 h = pack_bf16x4(v.x, v.y, v.z, v.w);
  const __nv_bfloat162 h01 = *reinterpret_cast<const __nv_bfloat162*>(&h.x);
  const __nv_bfloat162 h23 = *reinterpret_cast<const __nv_bfloat162*>(&h.y);
  const float2 f01 = __bfloat1622float2(h01), f23 = __bfloat1622float2(h23);
  *reinterpret_cast<uint2*>(d) = h;
  *reinterpret_cast<uint2*>(d + I) = pack_bf16x4(v.x - f01.x, v.y - f01.y, v.z - f23.x, v.w - f23.y);
  if (hi_again) *reinterpret_cast<uint2*>(d + 2 * I) = h;
}

// v = act(acc + b), acc rows of g groups of I columns (ld g I, I % 4 == 0): v as fp32
// (optional) and split (optional) at split[row][group][part][col] (ld parts g I): parts = 2
// stores hi, lo; parts = 3 stores hi, lo, hi
__global__ void bias_act_split(const float* __restrict__ acc, const float* __restrict__ b, int I, int g,
                               int64_t n, bool relu, float* __restrict__ out32,
                               __nv_bfloat16* __restrict__ split, int parts) {
  const int c = 4 * (blockIdx.x * blockDim.x + threadIdx.x);
  const int row_w = g * I;
  if (c >= row_w) return;
  const int gg = c / I, f = c - gg * I;
  const float4 bb = *reinterpret_cast<const float4*>(b + c);
  const int64_t step = row_step();
  for (int64_t r0 = row0(); r0 < n; r0 += kRowsPerThread * step) {
    float4 v[kRowsPerThread];
#pragma unroll
    for (int k = 0; k < kRowsPerThread; ++k)  // all loads first: several rows in flight
      if (r0 + k * step < n) v[k] = __ldcs(reinterpret_cast<const float4*>(acc + (r0 + k * step) * row_w + c));
#pragma unroll
    for (int k = 0; k < kRowsPerThread; ++k) {
      const int64_t r = r0 + k * step;
      if (r >= n) break;
      float4 x = v[k];
      x.x += bb.x; x.y += bb.y; x.z += bb.z; x.w += bb.w;
      if (relu) {
        x.x = fmaxf(x.x, 0.0f); x.y = fmaxf(x.y, 0.0f); x.z = fmaxf(x.z, 0.0f); x.w = fmaxf(x.w, 0.0f);
      }
      if (out32) *reinterpret_cast<float4*>(out32 + r * row_w + c) = x;
      if (split) store_split4(split + r * parts * row_w + (int64_t)gg * parts * I + f, I, x, parts == 3);
    }
  }
}

// x = lbar x (x = 0 first where reset) + Bbar u, in place; state [n][2P] (re, im), bu [n][2P];
// x also as [hi | lo | hi] bf16 rows of 2P each (ld 6P) for the three-term C product
__global__ void ssm_recur(const float* __restrict__ lbar, const float* __restrict__ bu,
                          const uint8_t* __restrict__ reset, float* __restrict__ state, int P,
                          int64_t n, __nv_bfloat16* __restrict__ xsplit) {
  const int p = 4 * (blockIdx.x * blockDim.x + threadIdx.x);
  if (p >= P) return;
  const float4 lr = *reinterpret_cast<const float4*>(lbar + p);
  const float4 li = *reinterpret_cast<const float4*>(lbar + P + p);
  for (int64_t e = row0(); e < n; e += row_step()) {
    float* s = state + e * 2 * P;
    const float* bp = bu + e * 2 * P;
    float4 xr = *reinterpret_cast<const float4*>(s + p), xi = *reinterpret_cast<const float4*>(s + P + p);
    if (reset[e]) xr = xi = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
    const float4 br = *reinterpret_cast<const float4*>(bp + p), bi = *reinterpret_cast<const float4*>(bp + P + p);
    float4 orr, oi;
    orr.x = fmaf(lr.x, xr.x, fmaf(-li.x, xi.x, br.x)); oi.x = fmaf(lr.x, xi.x, fmaf(li.x, xr.x, bi.x));
    orr.y = fmaf(lr.y, xr.y, fmaf(-li.y, xi.y, br.y)); oi.y = fmaf(lr.y, xi.y, fmaf(li.y, xr.y, bi.y));
    orr.z = fmaf(lr.z, xr.z, fmaf(-li.z, xi.z, br.z)); oi.z = fmaf(lr.z, xi.z, fmaf(li.z, xr.z, bi.z));
    orr.w = fmaf(lr.w, xr.w, fmaf(-li.w, xi.w, br.w)); oi.w = fmaf(lr.w, xi.w, fmaf(li.w, xr.w, bi.w));
    *reinterpret_cast<float4*>(s + p) = orr;
    *reinterpret_cast<float4*>(s + P + p) = oi;
    store_split4(xsplit + e * 6 * P + p, 2 * P, orr, true);
    store_split4(xsplit + e * 6 * P + P + p, 2 * P, oi, true);
  }
}

__device__ __forceinline__ float gelu_exact(float y) { return y * 0.5f * erfcf(-y * 0.70710678118654752f); }

// v = u + gelu(y + D u) -> split[row][0 | 1][H] (hi, lo bf16)
__global__ void residual_gelu(const float* __restrict__ y, const float* __restrict__ u,
                              const float* __restrict__ D, int H, int64_t n,
                              __nv_bfloat16* __restrict__ split) {
  const int c = 4 * (blockIdx.x * blockDim.x + threadIdx.x);
  if (c >= H) return;
  const float4 dd = *reinterpret_cast<const float4*>(D + c);
  for (int64_t r = row0(); r < n; r += row_step()) {
    const float4 uu = *reinterpret_cast<const float4*>(u + r * H + c);
    const float4 yy = *reinterpret_cast<const float4*>(y + r * H + c);
    float4 v;
    v.x = uu.x + gelu_exact(fmaf(dd.x, uu.x, yy.x));
    v.y = uu.y + gelu_exact(fmaf(dd.y, uu.y, yy.y));
    v.z = uu.z + gelu_exact(fmaf(dd.z, uu.z, yy.z));
    v.w = uu.w + gelu_exact(fmaf(dd.w, uu.w, yy.w));
    store_split4(split + r * 2 * H + c, H, v);
  }
}

__device__ __forceinline__ float warp_sum(float x) {
#pragma unroll
  for (int o = 16; o; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
  return x;
}

// The heads' last hidden layer and both output layers, one warp per env: h = relu(acc + b)
// in fp32 (acc [n][2F]: actor columns, then critic), logits[a] = Wa3[a] . h_actor + ba3[a]
// (-inf where illegal), value = Wc3 . h_critic + bc3. W3 [A + 1][F] fp32 (actor rows, then
// the critic's); AM >= A is the register width of the logit sums.
template <int AM>
__global__ void heads_out(const float* __restrict__ acc, const float* __restrict__ b,
                          const float* __restrict__ W3, const float* __restrict__ ba3,
                          const float* __restrict__ bc3, const uint8_t* __restrict__ legal, int A, int F,
                          int64_t n, float* __restrict__ logits, float* __restrict__ values) {
  const int lane = threadIdx.x & 31;
  const int64_t warps = (int64_t)gridDim.x * (blockDim.x >> 5);
  const int quads = F / 4;
  for (int64_t e = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); e < n; e += warps) {
    const float* row = acc + e * 2 * F;
    float pa[AM], pv = 0.0f;
#pragma unroll
    for (int a = 0; a < AM; ++a) pa[a] = 0.0f;
#pragma unroll 2
    for (int q = lane; q < quads; q += 32) {
      const float4 x = __ldcs(reinterpret_cast<const float4*>(row) + q);
      const float4 bb = reinterpret_cast<const float4*>(b)[q];
      const float4 h = make_float4(fmaxf(x.x + bb.x, 0.0f), fmaxf(x.y + bb.y, 0.0f), fmaxf(x.z + bb.z, 0.0f),
                                   fmaxf(x.w + bb.w, 0.0f));
#pragma unroll
      for (int a = 0; a < AM; ++a)
        if (a < A) {
          const float4 w = __ldg(reinterpret_cast<const float4*>(W3 + (size_t)a * F) + q);
          pa[a] = fmaf(h.x, w.x, fmaf(h.y, w.y, fmaf(h.z, w.z, fmaf(h.w, w.w, pa[a]))));
        }
      const float4 xc = __ldcs(reinterpret_cast<const float4*>(row + F) + q);
      const float4 bc = reinterpret_cast<const float4*>(b + F)[q];
      const float4 w = __ldg(reinterpret_cast<const float4*>(W3 + (size_t)A * F) + q);
      pv = fmaf(fmaxf(xc.x + bc.x, 0.0f), w.x, pv);
      pv = fmaf(fmaxf(xc.y + bc.y, 0.0f), w.y, pv);
      pv = fmaf(fmaxf(xc.z + bc.z, 0.0f), w.z, pv);
      pv = fmaf(fmaxf(xc.w + bc.w, 0.0f), w.w, pv);
    }
#pragma unroll
    for (int a = 0; a < AM; ++a)
      if (a < A) {
        const float z = warp_sum(pa[a]) + ba3[a];
        if (lane == a) logits[e * A + a] = (legal && !legal[e * A + a]) ? -INFINITY : z;
      }
    pv = warp_sum(pv);
    if (lane == 0) values[e] = pv + bc3[0];
  }
}

// launch shape of a row-wise kernel: 256 threads, x over a row's `quads` four-column groups
// (rounded up to a warp), y over rows; at most 65535 row blocks (the kernels stride)
struct RowsLaunch {
  dim3 grid, block;
};
RowsLaunch rows_launch(int quads, int64_t n, int rows_per_thread) {
  const int bx = std::min(256, (quads + 31) / 32 * 32), by = 256 / bx;
  const int64_t per_block = (int64_t)by * rows_per_thread;
  return {dim3((unsigned)((quads + bx - 1) / bx), (unsigned)std::min<int64_t>((n + per_block - 1) / per_block, 65535)),
          dim3((unsigned)bx, (unsigned)by)};
}
template <typename... KArgs, typename... Args>
void launch_rows(void (*kernel)(KArgs...), int quads, int64_t n, cudaStream_t st, Args... args) {
  const RowsLaunch L = rows_launch(quads, n, (void*)kernel == (void*)bias_act_split ? kRowsPerThread : 1);
  kernel<<<L.grid, L.block, 0, st>>>(args...);
}


// C[n][O] = X[n][I] W^T for row-major X (ld ldx), W [O][I] (ld I), C (ld ldc); `batch`
// products at once, the b-th at W + b sW, X + b sX, C + b sC
cublasStatus_t gemm_bf16(cublasHandle_t h, int64_t n, int O, int I, const __nv_bfloat16* W,
                         const __nv_bfloat16* X, int ldx, float* Cm, int ldc, int batch = 1,
                         int64_t sW = 0, int64_t sX = 0, int64_t sC = 0) {
  const float one = 1.0f, zero = 0.0f;
  if (batch == 1)
    return cublasGemmEx(h, CUBLAS_OP_T, CUBLAS_OP_N, O, (int)n, I, &one, W, CUDA_R_16BF, I, X, CUDA_R_16BF,
                        ldx, &zero, Cm, CUDA_R_32F, ldc, CUBLAS_COMPUTE_32F, CUBLAS_GEMM_DEFAULT);
  return cublasGemmStridedBatchedEx(h, CUBLAS_OP_T, CUBLAS_OP_N, O, (int)n, I, &one, W, CUDA_R_16BF, I, sW,
                                    X, CUDA_R_16BF, ldx, sX, &zero, Cm, CUDA_R_32F, ldc, sC, batch,
                                    CUBLAS_COMPUTE_32F, CUBLAS_GEMM_DEFAULT);
}

}  // namespace

extern "C" {

aht_status aht_s5_create(const aht_s5_params* p, int64_t max_envs, void* cuda_stream, aht_s5** out) {
  if (!out) return set_last_error(AHT_EINVAL, "out is NULL");
  *out = nullptr;
  if (!p) return set_last_error(AHT_EINVAL, "params is NULL");
  if (p->obs_dim < 1 || p->n_actions < 1 || p->n_actions > 32 || p->H < 16 || p->H % 16 || p->P < 16 ||
      p->P % 16 || p->F < 16 || p->F % 16)
    return set_last_error(AHT_EINVAL, "S5 sizes: obs_dim >= 1, 1 <= n_actions <= 32, H, P, F multiples of 16");
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
  s->Kp = (K + 15) / 16 * 16;
  s->max_n = max_envs;
  s->stream = static_cast<cudaStream_t>(cuda_stream);
  cudaGetDevice(&s->device);
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
  auto up16 = [&](__nv_bfloat16** dst, const std::vector<const float*>& parts, const std::vector<size_t>& counts) {
    size_t total = 0;
    for (size_t c : counts) total += c;
    std::vector<__nv_bfloat16> h(total);
    size_t o = 0;
    for (size_t k = 0; k < parts.size(); ++k)
      for (size_t i = 0; i < counts[k]; ++i) h[o++] = __float2bfloat16_rn(parts[k][i]);
    return alloc((void**)dst, total * 2) && cudaMemcpy(*dst, h.data(), total * 2, cudaMemcpyHostToDevice) == cudaSuccess;
  };
  auto up32 = [&](float** dst, const std::vector<float>& h) {
    return alloc((void**)dst, h.size() * 4) && cudaMemcpy(*dst, h.data(), h.size() * 4, cudaMemcpyHostToDevice) == cudaSuccess;
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
  // [W | W] rows: each of `rows` rows of every part written twice
  auto up16x2 = [&](__nv_bfloat16** dst, const std::vector<const float*>& parts, size_t rows, size_t cols) {
    std::vector<__nv_bfloat16> h(parts.size() * rows * 2 * cols);
    size_t o = 0;
    for (const float* w : parts)
      for (size_t r = 0; r < rows; ++r)
        for (int rep = 0; rep < 2; ++rep)
          for (size_t c = 0; c < cols; ++c) h[o++] = __float2bfloat16_rn(w[r * cols + c]);
    return alloc((void**)dst, h.size() * 2) && cudaMemcpy(*dst, h.data(), h.size() * 2, cudaMemcpyHostToDevice) == cudaSuccess;
  };
  std::vector<float> We1p((size_t)H * s->Kp, 0.0f);
  for (int h = 0; h < H; ++h) std::copy(p->We1 + (size_t)h * K, p->We1 + (size_t)(h + 1) * K, We1p.begin() + (size_t)h * s->Kp);
  bool ok = up16(&s->We1, {We1p.data()}, {We1p.size()}) && up16x2(&s->We2, {p->We2}, H, H) &&
            up16x2(&s->Wh0, {p->Wa[0], p->Wc[0]}, F, H) && up16x2(&s->Wh1, {p->Wa[1], p->Wc[1]}, F, F) &&
            up16x2(&s->Wh2, {p->Wa[2], p->Wc[2]}, F, F) &&
            up32(&s->W3, cat(bf16_rounded(p->Wa[3], (size_t)A * F), bf16_rounded(p->Wc[3], F))) &&
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
  // three-term bf16 rows [Wh | Wh | Wl] of an fp32 matrix [rows][cols]
  auto up_three = [&](__nv_bfloat16** dst, const std::vector<float>& w, size_t rows, size_t cols) {
    std::vector<__nv_bfloat16> h(rows * 3 * cols);
    for (size_t r = 0; r < rows; ++r)
      for (size_t c = 0; c < cols; ++c) {
        const float x = w[r * cols + c];
        const __nv_bfloat16 hi = __float2bfloat16_rn(x);
        h[r * 3 * cols + c] = hi;
        h[r * 3 * cols + cols + c] = hi;
        h[r * 3 * cols + 2 * cols + c] = __float2bfloat16_rn(x - __bfloat162float(hi));
      }
    return alloc((void**)dst, h.size() * 2) && cudaMemcpy(*dst, h.data(), h.size() * 2, cudaMemcpyHostToDevice) == cudaSuccess;
  };
  if (!up32(&s->lbar, lbar) || !up_three(&s->Bbar3, Bbar, 2 * P, H) || !up_three(&s->Cc3, Cc, H, 2 * P))
    return bail(AHT_ENOMEM, "S5 upload failed");
  const int64_t n = max_envs;
  ok = alloc((void**)&s->x16, (size_t)n * s->Kp * 2) && alloc((void**)&s->act, (size_t)n * std::max({4 * F, 3 * H, 6 * P}) * 2) &&
       alloc((void**)&s->acc, (size_t)n * std::max(2 * F, H) * 4) && alloc((void**)&s->u, (size_t)n * H * 4) &&
       alloc((void**)&s->bu, (size_t)n * 2 * P * 4) && alloc((void**)&s->y, (size_t)n * H * 4) &&
       alloc(&s->workspace, kWorkspace);
  if (!ok) return bail(AHT_ENOMEM, "S5 scratch allocation failed");
  if (cublasCreate(&s->blas) != CUBLAS_STATUS_SUCCESS || cublasSetStream(s->blas, s->stream) != CUBLAS_STATUS_SUCCESS ||
      cublasSetWorkspace(s->blas, s->workspace, kWorkspace) != CUBLAS_STATUS_SUCCESS ||
      cublasSetMathMode(s->blas, CUBLAS_DEFAULT_MATH) != CUBLAS_STATUS_SUCCESS)
    return bail(AHT_ECUDA, "cuBLAS set-up failed");
  *out = s;
  return AHT_OK;
}

void aht_s5_destroy(aht_s5* s) {
  if (!s) return;
  S5DeviceGuard g(s->device);
  if (s->blas) cublasDestroy(s->blas);
  for (void* q : s->owned) cudaFree(q);
  delete s;
}

aht_status aht_s5_step(aht_s5* s, const uint8_t* obs, const uint8_t* reset, const uint8_t* legal,
                       int64_t n, float* state, float* logits, float* values) {
  if (!s || !obs || !reset || !state || !logits || !values) return set_last_error(AHT_EINVAL, "NULL argument");
  if (n < 1 || n > s->max_n) return set_last_error(AHT_EINVAL, "n must be in 1..max_envs");
  S5DeviceGuard g(s->device);
  const int K = s->K, A = s->A, H = s->H, P = s->P, F = s->F;
  cudaStream_t st = s->stream;
  cublasHandle_t b = s->blas;
  // encoder: the observation is exact in bf16, so layer 1 is one plain product; later
  // layers take [hi | lo] against [W | W], one product with fp32 accumulation
  launch_rows(u8_to_bf16, s->Kp / 4, n, st, obs, s->x16, K, s->Kp, n);
  S5_BLAS(gemm_bf16(b, n, H, s->Kp, s->We1, s->x16, s->Kp, s->acc, H));
  launch_rows(bias_act_split, H / 4, n, st, s->acc, s->be1, H, 1, n, true, (float*)nullptr, s->act, 2);
  S5_BLAS(gemm_bf16(b, n, H, 2 * H, s->We2, s->act, 2 * H, s->acc, H));
  launch_rows(bias_act_split, H / 4, n, st, s->acc, s->be2, H, 1, n, true, s->u, s->act, 3);
  // SSM: Bbar u and Re(C x) as three-term bf16 products, the recurrence in fp32
  S5_BLAS(gemm_bf16(b, n, 2 * P, 3 * H, s->Bbar3, s->act, 3 * H, s->bu, 2 * P));
  launch_rows(ssm_recur, P / 4, n, st, s->lbar, s->bu, reset, state, P, n, s->act);
  S5_BLAS(gemm_bf16(b, n, H, 6 * P, s->Cc3, s->act, 6 * P, s->y, H));
  launch_rows(residual_gelu, H / 4, n, st, s->y, s->u, s->Dv, H, n, s->act);
  // heads: layer 0 for both heads at once ([2F] outputs, split as 2 groups of F), layers
  // 1-2 as one two-member batch (head h reads group h, writes columns h F of acc)
  S5_BLAS(gemm_bf16(b, n, 2 * F, 2 * H, s->Wh0, s->act, 2 * H, s->acc, 2 * F));
  launch_rows(bias_act_split, 2 * F / 4, n, st, s->acc, s->bh0, F, 2, n, true, (float*)nullptr, s->act, 2);
  const __nv_bfloat16* Wl[2] = {s->Wh1, s->Wh2};
  const float* bl[2] = {s->bh1, s->bh2};
  for (int l = 0; l < 2; ++l) {
    S5_BLAS(gemm_bf16(b, n, F, 2 * F, Wl[l], s->act, 4 * F, s->acc, 2 * F, 2, (int64_t)F * 2 * F, 2 * F, F));
    if (l == 0) launch_rows(bias_act_split, 2 * F / 4, n, st, s->acc, bl[l], F, 2, n, true, (float*)nullptr, s->act, 2);
  }
  // layer 2's bias and relu, and both output layers, in fp32 (one warp per env)
  const int out_blocks = (int)std::min<int64_t>((n + 7) / 8, 65535);
  if (A <= 8)
    heads_out<8><<<out_blocks, 256, 0, st>>>(s->acc, s->bh2, s->W3, s->ba3, s->bc3, legal, A, F, n, logits, values);
  else if (A <= 16)
    heads_out<16><<<out_blocks, 256, 0, st>>>(s->acc, s->bh2, s->W3, s->ba3, s->bc3, legal, A, F, n, logits, values);
  else
    heads_out<32><<<out_blocks, 256, 0, st>>>(s->acc, s->bh2, s->W3, s->ba3, s->bc3, legal, A, F, n, logits, values);
  S5_CUDA(cudaGetLastError());
  return AHT_OK;
}

aht_status aht_s5_sync(aht_s5* s) {
  if (!s) return set_last_error(AHT_EINVAL, "NULL argument");
  S5DeviceGuard g(s->device);
  S5_CUDA(cudaStreamSynchronize(s->stream));
  return AHT_OK;
}

}  // extern "C"
