// misc.cu -- env-independent kernels: teammate grouping, GAE, cross-play reduction and the
// standalone policy forward.
#include "kernels.h"
#include "mlp_simt.cuh"
#include "rollout_impl.cuh"
#include "tc_common.cuh"

namespace aht {

// ---- teammate assignment: one pool draw per block of kTeammateBlock envs ---------------
// Block k (envs 128k .. 128k+127) plays pool[floor(x * pool_size / 2^32)], x = first draw
// of (128k, step0, stream 3).  Tiles of up to M rows never cross a block, so each tile
// runs one teammate policy; the env order is the identity (perm[e] = e).
__global__ void group_kernel(const GroupArgs a) {
  const int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (e >= a.n_envs) return;
  const int64_t blk = e / kTeammateBlock, first = blk * kTeammateBlock;
  const uint32_t b = uniform_int(draw0(a.key, (uint32_t)first, a.step0, kStreamTeammate), (uint32_t)a.pool_size);
  const int tm = a.pool[b];
  a.perm[e] = (int32_t)e;
  if (a.teammate) a.teammate[e] = tm;
  if (e == first) {
    const int n_blk = (int)min((int64_t)kTeammateBlock, a.n_envs - first);
    const int tpb = (kTeammateBlock + a.M - 1) / a.M;
    for (int j = 0; j < tpb; ++j) {
      const int r0 = j * a.M, cnt = max(0, min(a.M, n_blk - r0));
      a.tiles[blk * tpb + j] = make_int4((int)first + r0, cnt, tm, 0);
    }
  }
}

int group_tiles(int64_t n_envs, int M) {
  return (int)(((n_envs + kTeammateBlock - 1) / kTeammateBlock) * ((kTeammateBlock + M - 1) / M));
}

cudaError_t launch_group(const GroupArgs& a, cudaStream_t s) {
  group_kernel<<<(unsigned)((a.n_envs + 255) / 256), 256, 0, s>>>(a);
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
  const int64_t i = 2 * (blockIdx.x * (int64_t)blockDim.x + threadIdx.x);  // elements i, i + 1
  if (i >= n) return;
  const float x1 = i + 1 < n ? x[i + 1] : 0.0f;
  float y0, y1;
  tc::f2_unpack(tc::tanh2(tc::f2_pack(x[i], x1)), y0, y1);
  y[i] = y0;
  if (i + 1 < n) y[i + 1] = y1;
}

// One thread waits on an mbarrier that nothing arrives on, with the kernels' bounded wait:
// the wait expires after limit_ns and the timeout bit is latched.
__global__ void expire_wait_kernel(uint32_t* status, uint64_t limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  tc::mbar_init(&bar, 1);
  tc::mbar_init_fence();
  if (!tc::mbar_wait(&bar, 0, limit_ns)) atomicOr(status, kStatusTimeout);
}

cudaError_t launch_expire_wait(uint32_t* status, uint64_t limit_ns, cudaStream_t s) {
  expire_wait_kernel<<<1, 1, 0, s>>>(status, limit_ns);
  return cudaGetLastError();
}

cudaError_t launch_tanh_probe(const float* x, float* y, int64_t n, cudaStream_t s) {
  const int64_t pairs = (n + 1) / 2;
  tanh_probe_kernel<<<(unsigned)((pairs + 255) / 256), 256, 0, s>>>(x, y, n);
  return cudaGetLastError();
}

}  // namespace aht
