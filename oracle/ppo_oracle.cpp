// ppo_oracle.cpp -- TEST INFRASTRUCTURE ONLY: the PPO ego update in fp64.
//
// App. C "PPO ego" trains the ego with PPO (Schulman et al. 2017) against the teammate
// distribution; the paper states no loss details or hyperparameters, so the update here
// is the clipped-surrogate PPO of that paper (policy term, clipped value term, entropy
// bonus), with per-minibatch advantage normalisation, global-norm gradient clipping and
// Adam (Kingma & Ba 2015), with the settings stated at orc_ppo_update in aht_oracle.h.  The
// forward and backward use bf16-rounded copies of W1 and W2 (the weights the bf16
// rollout runs), fp64 everywhere else; the gradient is taken at the rounded weights and
// applied to the fp64 master copy.  Plain loops in the order of the definitions.
#include <cmath>
#include <cstring>
#include <thread>
#include <vector>

#include "aht_oracle.h"

namespace {

// Round to bf16, nearest-even, through fp32 (the master copy the GPU keeps is fp32).
double bf16_of(double w) {
  float f = (float)w;
  uint32_t u;
  std::memcpy(&u, &f, 4);
  u = (u + 0x7FFFu + ((u >> 16) & 1u)) & 0xFFFF0000u;
  std::memcpy(&f, &u, 4);
  return (double)f;
}

int perm_bits(int64_t S) {
  int w = 2;
  while ((int64_t(1) << w) < S) ++w;
  return w;
}

// Four-round Feistel network on w-bit values (high half L, low half R); round r replaces
// one half by itself XOR a Philox word of the other half.
uint32_t feistel(uint64_t seed, uint32_t epoch, int w, uint32_t x) {
  const int rb = w / 2, lb = w - rb;
  const uint32_t rmask = (uint32_t)((1ull << rb) - 1), lmask = (uint32_t)((1ull << lb) - 1);
  uint32_t L = x >> rb, R = x & rmask;
  for (uint32_t r = 0; r < 4; ++r) {
    const uint32_t ctr[4] = {(r & 1u) ? L : R, epoch, (uint32_t)ORC_STREAM_PERMUTE, r};
    uint32_t o[4];
    orc_philox4x32_10((uint32_t)(seed & 0xffffffffu), (uint32_t)(seed >> 32), ctr, o);
    if ((r & 1u) == 0) L = (L ^ o[0]) & lmask;
    else R = (R ^ o[0]) & rmask;
  }
  return (L << rb) | R;
}

struct Offsets {
  int64_t W1, b1, W2, b2, W3, b3, total;
};
Offsets offsets(const orc_ppo_net* n) {
  const int64_t D = n->obs_dim, H0 = n->h0, H1 = n->h1, O = n->n_act + 1;
  Offsets o;
  o.W1 = 0;
  o.b1 = o.W1 + H0 * D;
  o.W2 = o.b1 + H0;
  o.b2 = o.W2 + H1 * H0;
  o.W3 = o.b2 + H1;
  o.b3 = o.W3 + O * H1;
  o.total = o.b3 + O;
  return o;
}

// Loss, its gradient and the diagnostics of one sample, added into grad/stats with
// weight 1/B.  Wq1/Wq2: the weights the forward uses.
void sample_grad(const orc_ppo_net* n, const Offsets& of, const double* p, const double* Wq1,
                 const double* Wq2, const orc_ppo_batch* tb, int64_t s, double mu, double sigma,
                 double B, const orc_ppo_hp* hp, double* grad, double* stats) {
  const int D = n->obs_dim, H0 = n->h0, H1 = n->h1, A = n->n_act, O = A + 1;
  std::vector<double> x(D), h1(H0), h2(H1), z(O), logp(A), prob(A), dz(O), dh2(H1), da2(H1),
      dh1(H0), da1(H0);
  for (int k = 0; k < D; ++k) x[k] = (double)tb->obs[s * D + k];
  // forward: h1 = tanh(W1 x + b1), h2 = tanh(W2 h1 + b2), z = W3 h2 + b3
  for (int o = 0; o < H0; ++o) {
    double acc = p[of.b1 + o];
    for (int k = 0; k < D; ++k) acc += Wq1[(int64_t)o * D + k] * x[k];
    h1[o] = std::tanh(acc);
  }
  for (int o = 0; o < H1; ++o) {
    double acc = p[of.b2 + o];
    for (int k = 0; k < H0; ++k) acc += Wq2[(int64_t)o * H0 + k] * h1[k];
    h2[o] = std::tanh(acc);
  }
  for (int j = 0; j < O; ++j) {
    double acc = p[of.b3 + j];
    for (int k = 0; k < H1; ++k) acc += p[of.W3 + (int64_t)j * H1 + k] * h2[k];
    z[j] = acc;
  }
  // log-softmax over the action logits, entropy
  double mx = z[0];
  for (int j = 1; j < A; ++j) mx = std::max(mx, z[j]);
  double se = 0.0;
  for (int j = 0; j < A; ++j) se += std::exp(z[j] - mx);
  const double lse = mx + std::log(se);
  double ent = 0.0;
  for (int j = 0; j < A; ++j) {
    logp[j] = z[j] - lse;
    prob[j] = std::exp(logp[j]);
    ent -= prob[j] * logp[j];
  }
  const int a = tb->actions[s];
  const double lp_old = (double)tb->logp[s], v_old = (double)tb->values[s];
  const double R = (double)tb->targets[s];
  const double adv = ((double)tb->advantages[s] - mu) / (sigma + 1e-8);
  const double eps = hp->clip_eps;
  // clipped surrogate: L_pg = -min(rho A, clip(rho, 1 - eps, 1 + eps) A)
  const double rho = std::exp(logp[a] - lp_old);
  const double rho_c = std::min(std::max(rho, 1.0 - eps), 1.0 + eps);
  const double un = rho * adv, cl = rho_c * adv;
  const double pg = -std::min(un, cl);
  const double g_rho = un <= cl ? -adv : 0.0;  // d L_pg / d rho (the clipped branch is flat)
  // clipped value loss: 0.5 max((V - R)^2, (V_old + clip(V - V_old, -eps, eps) - R)^2)
  const double V = z[A];
  const double vc = v_old + std::min(std::max(V - v_old, -eps), eps);
  const double u = V - R, w = vc - R;
  const double lv = 0.5 * std::max(u * u, w * w);
  const double dV = u * u >= w * w ? u : 0.0;  // a larger clipped branch has V outside the band
  const double loss = pg + hp->vf_coef * lv - hp->ent_coef * ent;
  // d loss / d z (mean over the minibatch)
  for (int j = 0; j < A; ++j) {
    const double dlogp = (j == a ? 1.0 : 0.0) - prob[j];
    const double dent = -prob[j] * (logp[j] + ent);  // d H / d z_j
    dz[j] = (g_rho * rho * dlogp - hp->ent_coef * dent) / B;
  }
  dz[A] = hp->vf_coef * dV / B;
  // backward
  for (int j = 0; j < O; ++j) {
    for (int k = 0; k < H1; ++k) grad[of.W3 + (int64_t)j * H1 + k] += dz[j] * h2[k];
    grad[of.b3 + j] += dz[j];
  }
  for (int k = 0; k < H1; ++k) {
    double acc = 0.0;
    for (int j = 0; j < O; ++j) acc += p[of.W3 + (int64_t)j * H1 + k] * dz[j];
    dh2[k] = acc;
    da2[k] = acc * (1.0 - h2[k] * h2[k]);
  }
  for (int o = 0; o < H1; ++o) {
    for (int k = 0; k < H0; ++k) grad[of.W2 + (int64_t)o * H0 + k] += da2[o] * h1[k];
    grad[of.b2 + o] += da2[o];
  }
  for (int k = 0; k < H0; ++k) {
    double acc = 0.0;
    for (int o = 0; o < H1; ++o) acc += Wq2[(int64_t)o * H0 + k] * da2[o];
    dh1[k] = acc;
    da1[k] = acc * (1.0 - h1[k] * h1[k]);
  }
  for (int o = 0; o < H0; ++o) {
    for (int k = 0; k < D; ++k) grad[of.W1 + (int64_t)o * D + k] += da1[o] * x[k];
    grad[of.b1 + o] += da1[o];
  }
  stats[0] += loss / B;
  stats[1] += pg / B;
  stats[2] += lv / B;
  stats[3] += ent / B;
  stats[4] += (lp_old - logp[a]) / B;
  stats[5] += (std::fabs(rho - 1.0) > eps ? 1.0 : 0.0) / B;
}

}  // namespace

extern "C" int64_t orc_ppo_n_params(const orc_ppo_net* n) { return offsets(n).total; }

extern "C" double orc_bf16_round(double w) { return bf16_of(w); }

extern "C" int64_t orc_perm_index(uint64_t seed, int64_t epoch, int64_t S, int64_t x) {
  const int w = perm_bits(S);
  uint32_t y = (uint32_t)x;
  do {
    y = feistel(seed, (uint32_t)epoch, w, y);
  } while ((int64_t)y >= S);
  return (int64_t)y;
}

extern "C" void orc_ppo_grad(const orc_ppo_net* n, const double* params, const orc_ppo_batch* tb,
                             const int64_t* idx, int64_t B, const orc_ppo_hp* hp, double* grad,
                             double* stats, int32_t n_threads) {
  const Offsets of = offsets(n);
  // the bf16 copies of W1 and W2 the forward runs (or the exact weights)
  std::vector<double> Wq1(params + of.W1, params + of.b1), Wq2(params + of.W2, params + of.b2);
  if (hp->round_bf16) {
    for (double& w : Wq1) w = bf16_of(w);
    for (double& w : Wq2) w = bf16_of(w);
  }
  // advantage normalisation over the minibatch: mean and population standard deviation
  double mu = 0.0;
  for (int64_t j = 0; j < B; ++j) mu += (double)tb->advantages[idx[j]];
  mu /= (double)B;
  double var = 0.0;
  for (int64_t j = 0; j < B; ++j) {
    const double d = (double)tb->advantages[idx[j]] - mu;
    var += d * d;
  }
  const double sigma = std::sqrt(var / (double)B);
  // per-thread partial sums over contiguous slices, added in thread order
  const int nt = n_threads < 1 ? 1 : n_threads;
  std::vector<std::vector<double>> g(nt, std::vector<double>(of.total, 0.0));
  std::vector<std::vector<double>> st(nt, std::vector<double>(6, 0.0));
  auto work = [&](int t) {
    const int64_t j0 = B * t / nt, j1 = B * (t + 1) / nt;
    for (int64_t j = j0; j < j1; ++j)
      sample_grad(n, of, params, Wq1.data(), Wq2.data(), tb, idx[j], mu, sigma, (double)B, hp,
                  g[t].data(), st[t].data());
  };
  std::vector<std::thread> th;
  for (int t = 1; t < nt; ++t) th.emplace_back(work, t);
  work(0);
  for (auto& x : th) x.join();
  for (int64_t i = 0; i < of.total; ++i) {
    double acc = 0.0;
    for (int t = 0; t < nt; ++t) acc += g[t][i];
    grad[i] = acc;
  }
  if (stats)
    for (int k = 0; k < 6; ++k) {
      double acc = 0.0;
      for (int t = 0; t < nt; ++t) acc += st[t][k];
      stats[k] = acc;
    }
}

extern "C" void orc_adam_step(int64_t n_params, double* params, double* m, double* v, int64_t* t,
                              double* grad, const orc_ppo_hp* hp) {
  // global-norm clipping: g * max / ||g|| when ||g|| >= max
  double sq = 0.0;
  for (int64_t i = 0; i < n_params; ++i) sq += grad[i] * grad[i];
  const double norm = std::sqrt(sq);
  if (hp->max_grad_norm > 0.0 && norm >= hp->max_grad_norm)
    for (int64_t i = 0; i < n_params; ++i) grad[i] = grad[i] / norm * hp->max_grad_norm;
  *t += 1;
  const double c1 = 1.0 - std::pow(hp->adam_b1, (double)*t);
  const double c2 = 1.0 - std::pow(hp->adam_b2, (double)*t);
  for (int64_t i = 0; i < n_params; ++i) {
    m[i] = hp->adam_b1 * m[i] + (1.0 - hp->adam_b1) * grad[i];
    v[i] = hp->adam_b2 * v[i] + (1.0 - hp->adam_b2) * grad[i] * grad[i];
    const double mh = m[i] / c1, vh = v[i] / c2;
    params[i] -= hp->lr * mh / (std::sqrt(vh) + hp->adam_eps);
  }
}

extern "C" void orc_ppo_update(const orc_ppo_net* n, double* params, double* m, double* v,
                               int64_t* t, const orc_ppo_batch* tb, int64_t S,
                               const orc_ppo_hp* hp, double* stats, int32_t n_threads) {
  const int64_t np = offsets(n).total;
  const int64_t B = S / hp->minibatches;
  std::vector<int64_t> perm(S);
  std::vector<double> grad(np);
  for (int e = 0; e < hp->epochs; ++e) {
    for (int64_t x = 0; x < S; ++x) perm[x] = orc_perm_index(hp->seed, hp->epoch0 + e, S, x);
    for (int b = 0; b < hp->minibatches; ++b) {
      double* st = stats ? stats + 6 * ((int64_t)e * hp->minibatches + b) : nullptr;
      orc_ppo_grad(n, params, tb, perm.data() + b * B, B, hp, grad.data(), st, n_threads);
      orc_adam_step(np, params, m, v, t, grad.data(), hp);
    }
  }
}
