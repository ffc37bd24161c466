// misc.cu -- env-independent kernels: teammate grouping, GAE, cross-play reduction and the
// standalone policy forward.
#include "kernels.h"
#include "mlp_simt.cuh"
#include "rollout_impl.cuh"
#include "tc_common.cuh"

namespace aht {

// ---- teammate assignment + stable grouping (one CTA) -----------------------------------
// Env e draws pool index b = floor(x * pool_size / 2^32), x = first draw of (e, step0,
// stream 3).  Envs are then ordered by b (stable in e) so that every tile of M rows
// shares one teammate policy.  cnt holds per-(bin, thread) counts, bin-major.
__global__ void __launch_bounds__(kGroupThreads) group_kernel(const GroupArgs a) {
  extern __shared__ uint32_t cnt[];  // [pool_size][kGroupThreads]
  __shared__ uint32_t seg[kGroupThreads];
  __shared__ uint32_t start[kMaxPool + 1];
  const int tid = threadIdx.x;
  const int P = a.pool_size;
  const int64_t chunk = (a.n_envs + kGroupThreads - 1) / kGroupThreads;
  const int64_t lo = tid * chunk, hi = min(a.n_envs, lo + chunk);
  for (int b = 0; b < P; ++b) cnt[b * kGroupThreads + tid] = 0;
  for (int64_t e = lo; e < hi; ++e) {
    const uint32_t b = uniform_int(draw0(a.key, (uint32_t)e, a.step0, kStreamTeammate), (uint32_t)P);
    cnt[b * kGroupThreads + tid] += 1;
  }
  __syncthreads();
  // Exclusive scan of the flattened counts: thread j owns entries [j*P, (j+1)*P).
  uint32_t run = 0;
  for (int q = 0; q < P; ++q) run += cnt[tid * P + q];
  seg[tid] = run;
  __syncthreads();
  if (tid == 0) {
    uint32_t acc = 0;
    for (int j = 0; j < kGroupThreads; ++j) {
      const uint32_t v = seg[j];
      seg[j] = acc;
      acc += v;
    }
  }
  __syncthreads();
  run = seg[tid];
  for (int q = 0; q < P; ++q) {
    const uint32_t v = cnt[tid * P + q];
    cnt[tid * P + q] = run;
    run += v;
  }
  __syncthreads();
  for (int b = tid; b <= P; b += blockDim.x) start[b] = b < P ? cnt[b * kGroupThreads] : (uint32_t)a.n_envs;
  __syncthreads();
  for (int64_t e = lo; e < hi; ++e) {
    const uint32_t b = uniform_int(draw0(a.key, (uint32_t)e, a.step0, kStreamTeammate), (uint32_t)P);
    const uint32_t pos = cnt[b * kGroupThreads + tid]++;
    a.perm[pos] = (int32_t)e;
    if (a.teammate) a.teammate[e] = a.pool[b];
  }
  if (tid == 0) {
    int t = 0;
    for (int b = 0; b < P; ++b) {
      const int n_b = (int)(start[b + 1] - start[b]);
      for (int j = 0; j * a.M < n_b; ++j)
        a.tiles[t++] = make_int4((int)start[b] + j * a.M, min(a.M, n_b - j * a.M), a.pool[b], 0);
    }
    for (; t < a.max_tiles; ++t) a.tiles[t] = make_int4(0, 0, 0, 0);
  }
}

size_t group_smem_bytes(int pool_size) { return (size_t)pool_size * kGroupThreads * 4; }

cudaError_t launch_group(const GroupArgs& a, cudaStream_t s) {
  const size_t smem = group_smem_bytes(a.pool_size);
  cudaError_t e = cudaFuncSetAttribute(group_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  group_kernel<<<1, kGroupThreads, smem, s>>>(a);
  return cudaGetLastError();
}

// ---- GAE: one thread per env, reverse scan over T (time-major, coalesced across envs) --
__global__ void gae_kernel(const float* __restrict__ r, const float* __restrict__ v,
                           const uint8_t* __restrict__ d, const float* __restrict__ v_last,
                           int64_t n, int32_t T, float gamma, float lambda,
                           float* __restrict__ adv, float* __restrict__ tgt) {
  const int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (e >= n) return;
  float next_v = v_last[e];
  float next_a = 0.0f;
  const float gl = gamma * lambda;
  for (int t = T - 1; t >= 0; --t) {
    const int64_t i = (int64_t)t * n + e;
    const float vt = v[i];
    const float nonterminal = d[i] ? 0.0f : 1.0f;
    const float delta = r[i] + gamma * nonterminal * next_v - vt;
    const float at = delta + gl * nonterminal * next_a;
    adv[i] = at;
    if (tgt) tgt[i] = at + vt;
    next_a = at;
    next_v = vt;
  }
}

cudaError_t launch_gae(const float* r, const float* v, const uint8_t* d, const float* v_last,
                       int64_t n, int32_t T, float gamma, float lambda, float* adv, float* tgt,
                       cudaStream_t s) {
  const int threads = 256;
  const int blocks = (int)((n + threads - 1) / threads);
  gae_kernel<<<blocks, threads, 0, s>>>(r, v, d, v_last, n, T, gamma, lambda, adv, tgt);
  return cudaGetLastError();
}

// ---- cross-play cell means: exact fp64 sum of each pair's P returns, divided by P -------
__global__ void xp_reduce_kernel(const float* __restrict__ returns, int32_t P,
                                 float* __restrict__ matrix) {
  __shared__ double part[256];
  const int64_t pair = blockIdx.x;
  double acc = 0.0;
  for (int k = threadIdx.x; k < P; k += blockDim.x) acc += (double)returns[pair * P + k];
  part[threadIdx.x] = acc;
  __syncthreads();
  for (int w = blockDim.x / 2; w > 0; w >>= 1) {
    if (threadIdx.x < w) part[threadIdx.x] += part[threadIdx.x + w];
    __syncthreads();
  }
  if (threadIdx.x == 0) matrix[pair] = (float)(part[0] / (double)P);
}

cudaError_t launch_xp_reduce(const float* returns, int64_t n_pairs, int32_t P, float* matrix,
                             cudaStream_t s) {
  xp_reduce_kernel<<<(unsigned)n_pairs, 256, 0, s>>>(returns, P, matrix);
  return cudaGetLastError();
}

// ---- standalone policy forward (test hook) ---------------------------------------------
__global__ void __launch_bounds__(kThreads) policy_kernel(const PolicyArgs a) {
  extern __shared__ __align__(16) uint8_t smem[];
  const MlpDims& m = a.b.mlp;
  const int M = a.M;
  const SmemLayout L = smem_layout(M, m, 0);
  uint8_t* X = smem + L.X;
  float* H1 = reinterpret_cast<float*>(smem + L.H1);
  float* H2 = reinterpret_cast<float*>(smem + L.H2);
  float* Z = reinterpret_cast<float*>(smem + L.Z);
  const int64_t r0 = (int64_t)blockIdx.x * M;
  const int count = (int)min((int64_t)M, a.n - r0);
  const int od = m.K;
  for (int idx = threadIdx.x; idx < M * m.KP; idx += blockDim.x) {
    const int i = idx / m.KP, k = idx - i * m.KP;
    X[idx] = (i < count && k < od) ? a.obs[(r0 + i) * od + k] : (uint8_t)0;
  }
  __syncthreads();
  mlp_tile(a.b.weights + (int64_t)a.policy * m.stride, m, X, H1, H2, Z, M);
  const int no = m.NA + 1;
  for (int idx = threadIdx.x; idx < count * no; idx += blockDim.x) {
    const int i = idx / no, c = idx - i * no;
    a.out[(r0 + i) * no + c] = Z[i * m.NOP + c];
  }
}

cudaError_t policy_set_smem_limit(size_t bytes) {
  return cudaFuncSetAttribute(policy_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
}

cudaError_t launch_policy(const PolicyArgs& a, int grid, size_t smem, cudaStream_t s) {
  policy_kernel<<<grid, kThreads, smem, s>>>(a);
  return cudaGetLastError();
}

// ---- the tensor-core epilogue's tanh, standalone (test hook) ---------------------------
__global__ void tanh_probe_kernel(const float* __restrict__ x, float* __restrict__ y, int64_t n) {
  const int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (i < n) y[i] = tc::tanh_ex2(x[i]);
}

cudaError_t launch_tanh_probe(const float* x, float* y, int64_t n, cudaStream_t s) {
  tanh_probe_kernel<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(x, y, n);
  return cudaGetLastError();
}

}  // namespace aht
