// misc.cu -- env-independent kernels: teammate grouping, GAE, cross-play reduction, the
// cross-play matrix consumers and the standalone policy forward.
#include <climits>

#include "kernels.h"
#include "mlp_simt.cuh"
#include "rollout_impl.cuh"
#include "tc_common.cuh"

namespace aht {

// ---- teammate assignment (Sec. 3: teammates drawn uniformly from the training pool) ----
// Per call, env e plays pool[floor(x * pool_size / 2^32)], x = first draw of (e, step0,
// stream 3), for the whole call.  With a one-member pool every env plays pool[0] (the
// draw is 0 whatever x is): group_kernel cuts the envs into contiguous tiles of up to M
// (perm[e] = e).  With a larger pool, teammate_draw_kernel writes each env's pool index
// and the envs per index; the tensor-core rollout then finds each tile's envs by a rank
// scan, and the CUDA-core path groups them with resample_group_kernel (per-call draw).
__global__ void group_kernel(const GroupArgs a) {
  const int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (e >= a.n_envs) return;
  const int tm = a.pool[0];
  a.perm[e] = (int32_t)e;
  if (a.teammate) a.teammate[e] = tm;
  if (e % a.M == 0) a.tiles[e / a.M] = make_int4((int)e, (int)min((int64_t)a.M, a.n_envs - e), tm, 0);
}

int group_tiles(int64_t n_envs, int M) { return (int)((n_envs + M - 1) / M); }

__global__ void teammate_draw_kernel(const GroupArgs a) {
  __shared__ int cnt[kMaxPool];
  const uint32_t P = (uint32_t)a.pool_size;
  for (int k = threadIdx.x; k < (int)P; k += blockDim.x) cnt[k] = 0;
  __syncthreads();
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < a.n_envs;
       e += (int64_t)gridDim.x * blockDim.x) {
    const uint32_t k = uniform_int(draw0(a.key, (uint32_t)e, a.step0, kStreamTeammate), P);
    a.kidx[e] = (uint8_t)k;
    if (a.teammate) a.teammate[e] = a.pool[k];
    atomicAdd(&cnt[k], 1);
  }
  __syncthreads();
  for (int k = threadIdx.x; k < (int)P; k += blockDim.x)
    if (cnt[k]) atomicAdd(&a.hist[k], cnt[k]);
}

cudaError_t launch_teammate_draw(const GroupArgs& a, cudaStream_t s) {
  int64_t blocks = (a.n_envs + 255) / 256;
  if (blocks > 148) blocks = 148;
  teammate_draw_kernel<<<(unsigned)blocks, 256, 0, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_group(const GroupArgs& a, cudaStream_t s) {
  group_kernel<<<(unsigned)((a.n_envs + 255) / 256), 256, 0, s>>>(a);
  return cudaGetLastError();
}

// ---- group the envs by their teammate's pool index (per episode, or per call) ----------
// One CTA: count the envs per pool index (shared-memory atomics), lay the groups out
// back to back in perm and cut each into tiles of up to M envs, then scatter the env ids.
// The order of the envs inside a group is not fixed (atomic slots); every row's result
// depends on its env id only.
__global__ void __launch_bounds__(1024) resample_group_kernel(const ResampleGroupArgs a) {
  __shared__ int cnt[kMaxPool], base[kMaxPool], tile0[kMaxPool];
  __shared__ int n_tiles;
  const int tid = threadIdx.x;
  const uint32_t P = (uint32_t)a.pool_size;
  // per episode: the draw of the step the env's episode began; per call (ep_step NULL):
  // the draw of the call's first step on the teammate stream
  auto index_of = [&](int64_t e) {
    return (int)uniform_int(a.ep_step ? draw0(a.key, (uint32_t)e, a.ep_step[e], kStreamEpisodeTeammate)
                                      : draw0(a.key, (uint32_t)e, a.step0, kStreamTeammate),
                            P);
  };
  for (int k = tid; k < a.pool_size; k += blockDim.x) cnt[k] = 0;
  __syncthreads();
  for (int64_t e = tid; e < a.n_envs; e += blockDim.x) atomicAdd(&cnt[index_of(e)], 1);
  __syncthreads();
  if (tid == 0) {
    int off = 0, t = 0;
    for (int k = 0; k < a.pool_size; ++k) {
      base[k] = off;
      tile0[k] = t;
      off += cnt[k];
      t += (cnt[k] + a.M - 1) / a.M;
    }
    n_tiles = t;
  }
  __syncthreads();
  for (int k = tid; k < a.pool_size; k += blockDim.x) {
    const int n = cnt[k];
    for (int j = 0; j * a.M < n; ++j)
      a.tiles[tile0[k] + j] = make_int4(base[k] + j * a.M, min(a.M, n - j * a.M), a.pool[k], 0);
  }
  for (int j = n_tiles + tid; j < a.max_tiles; j += blockDim.x) a.tiles[j] = make_int4(0, 0, 0, 0);
  __syncthreads();
  for (int k = tid; k < a.pool_size; k += blockDim.x) cnt[k] = base[k];  // slot cursors
  __syncthreads();
  for (int64_t e = tid; e < a.n_envs; e += blockDim.x) {
    const int k = index_of(e);
    a.perm[atomicAdd(&cnt[k], 1)] = (int32_t)e;
    if (a.teammate) a.teammate[e] = a.pool[k];
    if (a.teammate2) a.teammate2[e] = a.pool[k];
  }
}

__global__ void resample_init_kernel(const Key key, int64_t n, const uint32_t* __restrict__ ep_step,
                                     uint32_t P, uint8_t* __restrict__ kidx, int32_t* __restrict__ hist) {
  __shared__ int cnt[kMaxPool];
  for (int k = threadIdx.x; k < (int)P; k += blockDim.x) cnt[k] = 0;
  __syncthreads();
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < n; e += (int64_t)gridDim.x * blockDim.x) {
    const uint32_t k = uniform_int(draw0(key, (uint32_t)e, ep_step[e], kStreamEpisodeTeammate), P);
    kidx[e] = (uint8_t)k;
    atomicAdd(&cnt[k], 1);
  }
  __syncthreads();
  for (int k = threadIdx.x; k < (int)P; k += blockDim.x)
    if (cnt[k]) atomicAdd(&hist[k], cnt[k]);
}

cudaError_t launch_resample_init(const Key& key, int64_t n_envs, const uint32_t* ep_step,
                                 int32_t pool_size, uint8_t* kidx, int32_t* hist, cudaStream_t s) {
  int64_t blocks = (n_envs + 255) / 256;
  if (blocks > 148) blocks = 148;
  resample_init_kernel<<<(unsigned)blocks, 256, 0, s>>>(key, n_envs, ep_step, (uint32_t)pool_size, kidx, hist);
  return cudaGetLastError();
}

int resample_tiles(int64_t n_envs, int M, int pool_size) {
  return (int)((n_envs + M - 1) / M) + pool_size;
}

cudaError_t launch_resample_group(const ResampleGroupArgs& a, cudaStream_t s) {
  resample_group_kernel<<<1, 1024, 0, s>>>(a);
  return cudaGetLastError();
}

// ---- GAE: one thread per env, reverse scan over T (time-major, coalesced across envs) --
// The scan carries only two floats from step to step, so each thread loads the rewards,
// values and done flags of kGaeChunk steps at once (independent loads in flight together)
// and then runs the recurrence over them in the same order as a step-by-step scan.
constexpr int kGaeChunk = 16;

__global__ void __launch_bounds__(128) gae_kernel(const float* __restrict__ r, const float* __restrict__ v,
                                                  const uint8_t* __restrict__ d, const float* __restrict__ v_last,
                                                  int64_t n, int32_t T, float gamma, float lambda,
                                                  float* __restrict__ adv, float* __restrict__ tgt) {
  // launched as a programmatic dependent of the stream's previous kernel (the rollout
  // that wrote the trajectory): wait until it is complete
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (e >= n) return;
  float next_v = v_last[e];
  float next_a = 0.0f;
  const float gl = gamma * lambda;
  for (int t0 = T - 1; t0 >= 0; t0 -= kGaeChunk) {
    const int c = t0 + 1 < kGaeChunk ? t0 + 1 : kGaeChunk;  // steps t0, t0 - 1, ..., t0 - c + 1
    float rv[kGaeChunk], vv[kGaeChunk];
    uint8_t dv[kGaeChunk];
#pragma unroll
    for (int j = 0; j < kGaeChunk; ++j)
      if (j < c) {
        const int64_t i = (int64_t)(t0 - j) * n + e;
        rv[j] = r[i];
        vv[j] = v[i];
        dv[j] = d[i];
      }
#pragma unroll
    for (int j = 0; j < kGaeChunk; ++j)
      if (j < c) {
        const int64_t i = (int64_t)(t0 - j) * n + e;
        const float nonterminal = dv[j] ? 0.0f : 1.0f;
        const float delta = rv[j] + gamma * nonterminal * next_v - vv[j];
        const float at = delta + gl * nonterminal * next_a;
        adv[i] = at;
        if (tgt) tgt[i] = at + vv[j];
        next_a = at;
        next_v = vv[j];
      }
  }
}

cudaError_t launch_gae(const float* r, const float* v, const uint8_t* d, const float* v_last,
                       int64_t n, int32_t T, float gamma, float lambda, float* adv, float* tgt,
                       cudaStream_t s) {
  const int threads = 128;  // 16384 envs -> 128 CTAs, spread over the SMs
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)((n + threads - 1) / threads));
  cfg.blockDim = dim3(threads);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, gae_kernel, r, v, d, v_last, n, T, gamma, lambda, adv, tgt);
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

// ---- cross-play matrix consumers -------------------------------------------------------
// xp [n_ego][n_tm]: rows are the policies in the ego seat (best responses, or the ego),
// columns the evaluation teammates.  App. B "Upper bound estimation": each teammate's
// recorded bound is raised to any cross-play score that exceeds it.  Returns are reported
// relative to that bound (Sec. 3, the best response's return); J_AHT is the row mean
// (Sec. 3, teammates uniform); the cooperative regret is bound minus return (App. A,
// ROTATE); BRDiv's cross-play objective is the matched (diagonal) mean minus the
// mismatched mean (App. A).  One CTA of 1024 threads: a thread per column for the bounds
// (rows in order), then a warp per row -- lanes take every 32nd column, in fp64, and the
// row's sums and its largest regret are combined by shuffles -- then warp 0 for the BRDiv
// sums.  FP64 is slow on this part, so the divisions run across lanes, not in a chain.
constexpr int kXpStatsThreads = 1024;

__device__ __forceinline__ double warp_sum_f64(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = __dadd_rn(v, __shfl_xor_sync(0xFFFFFFFFu, v, o));
  return v;
}

__global__ void __launch_bounds__(kXpStatsThreads) xp_stats_kernel(const XpStatsArgs a) {
  __shared__ float up[kXpStatsMax];
  __shared__ double off_row[kXpStatsMax];
  const int ne = a.n_ego, nt = a.n_tm;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, n_warps = blockDim.x >> 5;
  for (int m = threadIdx.x; m < nt; m += blockDim.x) {
    float u = a.upper[m];
    for (int e = 0; e < ne; ++e) {
      const float x = a.xp[(int64_t)e * nt + m];
      if (x > u) u = x;  // strict: a NaN bound is never exceeded
    }
    up[m] = u;
    a.upper[m] = u;
  }
  __syncthreads();
  const double nan = __longlong_as_double(0x7FF8000000000000ll);
  for (int e = warp; e < ne; e += n_warps) {
    double sum = 0.0, sum_norm = 0.0, off = 0.0, best = -INFINITY;
    int arg = INT_MAX;  // this lane's largest non-NaN regret, its first column
    for (int m = lane; m < nt; m += 32) {
      const int64_t i = (int64_t)e * nt + m;
      const double x = (double)a.xp[i], u = (double)up[m];
      const double nr = u > 0.0 ? __ddiv_rn(x, u) : nan;
      const double rg = __dsub_rn(u, x);
      if (a.norm) a.norm[i] = __double2float_rn(nr);
      if (a.regret) a.regret[i] = __double2float_rn(rg);
      sum = __dadd_rn(sum, x);
      sum_norm = __dadd_rn(sum_norm, nr);
      if (rg > best) {
        best = rg;
        arg = m;
      }
      if (m != e) off = __dadd_rn(off, x);
    }
    sum = warp_sum_f64(sum);
    sum_norm = warp_sum_f64(sum_norm);
    off = warp_sum_f64(off);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const double ob = __shfl_xor_sync(0xFFFFFFFFu, best, o);
      const int oa = __shfl_xor_sync(0xFFFFFFFFu, arg, o);
      if (ob > best || (ob == best && oa < arg)) {
        best = ob;
        arg = oa;
      }
    }
    if (lane == 0) {
      // the scan's reading: start at column 0 and move on to strictly larger regrets, so
      // a NaN at column 0 stays (the bound of teammate 0 is NaN) and later NaNs never win
      const double rg0 = __dsub_rn((double)up[0], (double)a.xp[(int64_t)e * nt]);
      if (rg0 != rg0 || arg == INT_MAX) {
        best = rg0;
        arg = 0;
      }
      if (a.j_aht) a.j_aht[e] = __double2float_rn(__ddiv_rn(sum, (double)nt));
      if (a.j_norm) a.j_norm[e] = __double2float_rn(__ddiv_rn(sum_norm, (double)nt));
      if (a.max_regret) a.max_regret[e] = __double2float_rn(best);
      if (a.worst) a.worst[e] = arg;
      off_row[e] = off;
    }
  }
  __syncthreads();
  if (warp == 0 && a.brdiv && ne == nt) {
    double diag = 0.0, off = 0.0;
    for (int i = lane; i < ne; i += 32) {
      diag = __dadd_rn(diag, (double)a.xp[(int64_t)i * nt + i]);
      off = __dadd_rn(off, off_row[i]);
    }
    diag = warp_sum_f64(diag);
    off = warp_sum_f64(off);
    if (lane == 0) {
      const double mis = ne > 1 ? __ddiv_rn(off, (double)ne * (double)(ne - 1)) : 0.0;
      *a.brdiv = __double2float_rn(__dsub_rn(__ddiv_rn(diag, (double)ne), mis));
    }
  }
}

cudaError_t launch_xp_stats(const XpStatsArgs& a, cudaStream_t s) {
  xp_stats_kernel<<<1, kXpStatsThreads, 0, s>>>(a);
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
  mlp_tile(a.b.weights + (int64_t)a.policy * m.stride, m, X, H1, H2, Z, M,
           reinterpret_cast<uint32_t*>(smem + L.list), count);
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
