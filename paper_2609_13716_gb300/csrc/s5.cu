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

struct aht_s5 {
  int device = 0;
  cudaStream_t stream = nullptr;
  cublasHandle_t blas = nullptr;
  int K = 0, A = 0, H = 0, P = 0, F = 0;
  int64_t max_n = 0;
  // bf16 weights [out][in]; heads stacked: layer 0 [2F][H] (actor rows, then critic),
  // layers 1-2 [2][F][F], layer 3 actor [A][F] and critic [1][F]
  __nv_bfloat16 *We1 = nullptr, *We2 = nullptr, *Wh0 = nullptr, *Wh1 = nullptr, *Wh2 = nullptr,
                *Wa3 = nullptr, *Wc3 = nullptr;
  float *be1 = nullptr, *be2 = nullptr, *bh0 = nullptr, *bh1 = nullptr, *bh2 = nullptr,
        *ba3 = nullptr, *bc3 = nullptr;
  // SSM: lbar [2][P] (re, im), Bbar [2P][H] (re rows, then im rows), Cc [H][2P] (C_re | -C_im), D [H]
  float *lbar = nullptr, *Bbar = nullptr, *Cc = nullptr, *Dv = nullptr;
  // scratch
  __nv_bfloat16 *x16 = nullptr, *hi = nullptr, *lo = nullptr;  // [n][K], [n][2F] each
  float *acc = nullptr, *u = nullptr, *bu = nullptr, *xs = nullptr, *y = nullptr;
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

__global__ void u8_to_bf16(const uint8_t* __restrict__ in, __nv_bfloat16* __restrict__ out, int64_t n) {
  const int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (i < n) out[i] = __float2bfloat16_rn((float)in[i]);
}

// out = act(acc + b) as fp32 (optional) and as hi + lo bf16, rows of `cols` (ld = cols)
__global__ void bias_act_split(const float* __restrict__ acc, const float* __restrict__ b, int cols,
                               int64_t total, bool relu, float* __restrict__ out32,
                               __nv_bfloat16* __restrict__ hi, __nv_bfloat16* __restrict__ lo) {
  const int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (i >= total) return;
  float v = acc[i] + b[i % cols];
  if (relu) v = fmaxf(v, 0.0f);
  if (out32) out32[i] = v;
  const __nv_bfloat16 h = __float2bfloat16_rn(v);
  hi[i] = h;
  lo[i] = __float2bfloat16_rn(v - __bfloat162float(h));
}

// x = lbar x (x = 0 first where reset) + Bbar u; state [n][2P], bu [n][2P], xs = state out
__global__ void ssm_recur(const float* __restrict__ lbar, const float* __restrict__ bu,
                          const uint8_t* __restrict__ reset, float* __restrict__ state, int P,
                          int64_t n) {
  const int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (i >= n * P) return;
  const int64_t e = i / P;
  const int p = (int)(i - e * P);
  float* s = state + e * 2 * P;
  const float xr = reset[e] ? 0.0f : s[p], xi = reset[e] ? 0.0f : s[P + p];
  const float lr = lbar[p], li = lbar[P + p];
  const float* b = bu + e * 2 * P;
  s[p] = fmaf(lr, xr, fmaf(-li, xi, b[p]));
  s[P + p] = fmaf(lr, xi, fmaf(li, xr, b[P + p]));
}

// v = u + gelu(y + D u) -> hi + lo bf16
__global__ void residual_gelu(const float* __restrict__ y, const float* __restrict__ u,
                              const float* __restrict__ D, int H, int64_t total,
                              __nv_bfloat16* __restrict__ hi, __nv_bfloat16* __restrict__ lo) {
  const int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (i >= total) return;
  const float uu = u[i];
  const float yy = fmaf(D[i % H], uu, y[i]);
  const float v = uu + yy * 0.5f * erfcf(-yy * 0.70710678118654752f);
  const __nv_bfloat16 h = __float2bfloat16_rn(v);
  hi[i] = h;
  lo[i] = __float2bfloat16_rn(v - __bfloat162float(h));
}

// logits = acc_a + ba (-inf where illegal), value = acc_c + bc
__global__ void s5_outputs(const float* __restrict__ acc_a, const float* __restrict__ acc_c,
                           const float* __restrict__ ba, const float* __restrict__ bc,
                           const uint8_t* __restrict__ legal, int A, int64_t n,
                           float* __restrict__ logits, float* __restrict__ values) {
  const int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (i < n * A) {
    const int a = (int)(i % A);
    const float z = acc_a[i] + ba[a];
    logits[i] = (legal && !legal[i]) ? -INFINITY : z;
  }
  if (i < n) values[i] = acc_c[i] + bc[0];
}

int blocks_for(int64_t total) { return (int)((total + 255) / 256); }

// C[n][O] (+)= X[n][I] W^T for row-major X (ld ldx), W [O][I] (ld I), C (ld ldc)
cublasStatus_t gemm_bf16(cublasHandle_t h, int64_t n, int O, int I, const __nv_bfloat16* W,
                         const __nv_bfloat16* X, int ldx, float* Cm, int ldc, float beta) {
  const float one = 1.0f;
  return cublasGemmEx(h, CUBLAS_OP_T, CUBLAS_OP_N, O, (int)n, I, &one, W, CUDA_R_16BF, I, X, CUDA_R_16BF,
                      ldx, &beta, Cm, CUDA_R_32F, ldc, CUBLAS_COMPUTE_32F, CUBLAS_GEMM_DEFAULT);
}
cublasStatus_t gemm_f32(cublasHandle_t h, int64_t n, int O, int I, const float* W, const float* X,
                        float* Cm) {
  const float one = 1.0f, zero = 0.0f;
  return cublasGemmEx(h, CUBLAS_OP_T, CUBLAS_OP_N, O, (int)n, I, &one, W, CUDA_R_32F, I, X, CUDA_R_32F, I,
                      &zero, Cm, CUDA_R_32F, O, CUBLAS_COMPUTE_32F, CUBLAS_GEMM_DEFAULT);
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
  auto cat = [](std::vector<float> a, const std::vector<float>& b) {
    a.insert(a.end(), b.begin(), b.end());
    return a;
  };
  bool ok = up16(&s->We1, {p->We1}, {(size_t)H * K}) && up16(&s->We2, {p->We2}, {(size_t)H * H}) &&
            up16(&s->Wh0, {p->Wa[0], p->Wc[0]}, {(size_t)F * H, (size_t)F * H}) &&
            up16(&s->Wh1, {p->Wa[1], p->Wc[1]}, {(size_t)F * F, (size_t)F * F}) &&
            up16(&s->Wh2, {p->Wa[2], p->Wc[2]}, {(size_t)F * F, (size_t)F * F}) &&
            up16(&s->Wa3, {p->Wa[3]}, {(size_t)A * F}) && up16(&s->Wc3, {p->Wc[3]}, {(size_t)F}) &&
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
  if (!up32(&s->lbar, lbar) || !up32(&s->Bbar, Bbar) || !up32(&s->Cc, Cc)) return bail(AHT_ENOMEM, "S5 upload failed");
  const int64_t n = max_envs;
  const int widest = std::max(2 * F, std::max(2 * P, H));
  ok = alloc((void**)&s->x16, (size_t)n * K * 2) && alloc((void**)&s->hi, (size_t)n * widest * 2) &&
       alloc((void**)&s->lo, (size_t)n * widest * 2) && alloc((void**)&s->acc, (size_t)n * widest * 4) &&
       alloc((void**)&s->u, (size_t)n * H * 4) && alloc((void**)&s->bu, (size_t)n * 2 * P * 4) &&
       alloc((void**)&s->y, (size_t)n * (2 * F > H ? 2 * F : H) * 4) && alloc(&s->workspace, kWorkspace);
  if (!ok) return bail(AHT_ENOMEM, "S5 scratch allocation failed");
  if (cublasCreate(&s->blas) != CUBLAS_STATUS_SUCCESS || cublasSetStream(s->blas, s->stream) != CUBLAS_STATUS_SUCCESS ||
      cublasSetWorkspace(s->blas, s->workspace, kWorkspace) != CUBLAS_STATUS_SUCCESS ||
      cublasSetMathMode(s->blas, CUBLAS_PEDANTIC_MATH) != CUBLAS_STATUS_SUCCESS)
    return bail(AHT_ECUDA, "cuBLAS set-up failed");
  *out = s;
  return AHT_OK;
}

void aht_s5_destroy(aht_s5* s) {
  if (!s) return;
  if (s->blas) cublasDestroy(s->blas);
  for (void* q : s->owned) cudaFree(q);
  delete s;
}

aht_status aht_s5_step(aht_s5* s, const uint8_t* obs, const uint8_t* reset, const uint8_t* legal,
                       int64_t n, float* state, float* logits, float* values) {
  if (!s || !obs || !reset || !state || !logits || !values) return set_last_error(AHT_EINVAL, "NULL argument");
  if (n < 1 || n > s->max_n) return set_last_error(AHT_EINVAL, "n must be in 1..max_envs");
  const int K = s->K, A = s->A, H = s->H, P = s->P, F = s->F;
  cudaStream_t st = s->stream;
  cublasHandle_t b = s->blas;
  // encoder: the observation is exact in bf16, so layer 1 is one product
  u8_to_bf16<<<blocks_for(n * K), 256, 0, st>>>(obs, s->x16, n * K);
  S5_BLAS(gemm_bf16(b, n, H, K, s->We1, s->x16, K, s->acc, H, 0.0f));
  bias_act_split<<<blocks_for(n * H), 256, 0, st>>>(s->acc, s->be1, H, n * H, true, nullptr, s->hi, s->lo);
  S5_BLAS(gemm_bf16(b, n, H, H, s->We2, s->hi, H, s->acc, H, 0.0f));
  S5_BLAS(gemm_bf16(b, n, H, H, s->We2, s->lo, H, s->acc, H, 1.0f));
  bias_act_split<<<blocks_for(n * H), 256, 0, st>>>(s->acc, s->be2, H, n * H, true, s->u, s->hi, s->lo);
  // SSM (fp32): Bbar u, the recurrence, Re(C x)
  S5_BLAS(gemm_f32(b, n, 2 * P, H, s->Bbar, s->u, s->bu));
  ssm_recur<<<blocks_for(n * P), 256, 0, st>>>(s->lbar, s->bu, reset, state, P, n);
  S5_BLAS(gemm_f32(b, n, H, 2 * P, s->Cc, state, s->y));
  residual_gelu<<<blocks_for(n * H), 256, 0, st>>>(s->y, s->u, s->Dv, H, n * H, s->hi, s->lo);
  // heads: layer 0 for both heads at once ([2F] outputs), layers 1-2 per head
  S5_BLAS(gemm_bf16(b, n, 2 * F, H, s->Wh0, s->hi, H, s->acc, 2 * F, 0.0f));
  S5_BLAS(gemm_bf16(b, n, 2 * F, H, s->Wh0, s->lo, H, s->acc, 2 * F, 1.0f));
  bias_act_split<<<blocks_for(n * 2 * F), 256, 0, st>>>(s->acc, s->bh0, 2 * F, n * 2 * F, true, nullptr, s->hi, s->lo);
  const __nv_bfloat16* Wl[2] = {s->Wh1, s->Wh2};
  const float* bl[2] = {s->bh1, s->bh2};
  for (int l = 0; l < 2; ++l) {
    for (int head = 0; head < 2; ++head) {
      const __nv_bfloat16* Wh = Wl[l] + (size_t)head * F * F;
      S5_BLAS(gemm_bf16(b, n, F, F, Wh, s->hi + head * F, 2 * F, s->acc + head * F, 2 * F, 0.0f));
      S5_BLAS(gemm_bf16(b, n, F, F, Wh, s->lo + head * F, 2 * F, s->acc + head * F, 2 * F, 1.0f));
    }
    bias_act_split<<<blocks_for(n * 2 * F), 256, 0, st>>>(s->acc, bl[l], 2 * F, n * 2 * F, true, nullptr, s->hi, s->lo);
  }
  // output layers: actor logits [n][A] into acc, critic value [n] into y
  S5_BLAS(gemm_bf16(b, n, A, F, s->Wa3, s->hi, 2 * F, s->acc, A, 0.0f));
  S5_BLAS(gemm_bf16(b, n, A, F, s->Wa3, s->lo, 2 * F, s->acc, A, 1.0f));
  S5_BLAS(gemm_bf16(b, n, 1, F, s->Wc3, s->hi + F, 2 * F, s->y, 1, 0.0f));
  S5_BLAS(gemm_bf16(b, n, 1, F, s->Wc3, s->lo + F, 2 * F, s->y, 1, 1.0f));
  s5_outputs<<<blocks_for(n * A), 256, 0, st>>>(s->acc, s->y, s->ba3, s->bc3, legal, A, n, logits, values);
  S5_CUDA(cudaGetLastError());
  return AHT_OK;
}

aht_status aht_s5_sync(aht_s5* s) {
  if (!s) return set_last_error(AHT_EINVAL, "NULL argument");
  S5_CUDA(cudaStreamSynchronize(s->stream));
  return AHT_OK;
}

}  // extern "C"
