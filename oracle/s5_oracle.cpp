// s5_oracle.cpp -- fp64 reference of the recurrent S5 actor-critic (the readings are in
// aht_oracle.h).  Test infrastructure only: the tests and the bench's CPU baseline call
// it, the library never does.  Plain loops in the order of the definitions.
#include <cmath>
#include <complex>
#include <thread>
#include <vector>

#include "aht_oracle.h"

namespace {

using cplx = std::complex<double>;

double relu(double a) { return a > 0.0 ? a : 0.0; }
double gelu(double a) { return a * 0.5 * std::erfc(-a / std::sqrt(2.0)); }

// out[r] = b[r] + sum_k W[r][k] in[k]
void dense(const double* W, const double* b, const double* in, int rows, int cols, double* out) {
  for (int r = 0; r < rows; ++r) {
    double acc = b[r];
    for (int k = 0; k < cols; ++k) acc += W[(size_t)r * cols + k] * in[k];
    out[r] = acc;
  }
}

}  // namespace

extern "C" void orc_s5_encode(const orc_s5_net* n, const uint8_t* obs, double* u) {
  std::vector<double> x(n->obs_dim), e1(n->H);
  for (int k = 0; k < n->obs_dim; ++k) x[k] = obs[k];
  dense(n->We1, n->be1, x.data(), n->H, n->obs_dim, e1.data());
  for (double& a : e1) a = relu(a);
  dense(n->We2, n->be2, e1.data(), n->H, n->H, u);
  for (int h = 0; h < n->H; ++h) u[h] = relu(u[h]);
}

extern "C" void orc_s5_ssm_step(const orc_s5_net* n, const double* u, int32_t reset, double* state,
                                double* y) {
  const int P = n->P, H = n->H;
  if (reset)
    for (int i = 0; i < 2 * P; ++i) state[i] = 0.0;
  std::vector<cplx> x(P);
  for (int p = 0; p < P; ++p) {
    const cplx lam(n->lam_re[p], n->lam_im[p]);
    const double dt = std::exp(n->log_dt[p]);
    const cplx lbar = std::exp(lam * dt);
    const cplx scale = (lbar - 1.0) / lam;
    cplx bu = 0.0;
    for (int h = 0; h < H; ++h) bu += cplx(n->B_re[(size_t)p * H + h], n->B_im[(size_t)p * H + h]) * u[h];
    x[p] = lbar * cplx(state[p], state[P + p]) + scale * bu;
    state[p] = x[p].real();
    state[P + p] = x[p].imag();
  }
  for (int h = 0; h < H; ++h) {
    cplx acc = 0.0;
    for (int p = 0; p < P; ++p) acc += cplx(n->C_re[(size_t)h * P + p], n->C_im[(size_t)h * P + p]) * x[p];
    y[h] = acc.real() + n->Dv[h] * u[h];
  }
}

extern "C" void orc_s5_heads(const orc_s5_net* n, const double* v, const uint8_t* legal,
                             double* logits, double* value) {
  const int F = n->F, H = n->H, A = n->n_actions;
  std::vector<double> a(F), b(F);
  for (int head = 0; head < 2; ++head) {
    const double* const* W = head == 0 ? n->Wa : n->Wc;
    const double* const* bb = head == 0 ? n->ba : n->bc;
    dense(W[0], bb[0], v, F, H, a.data());
    for (double& t : a) t = relu(t);
    dense(W[1], bb[1], a.data(), F, F, b.data());
    for (double& t : b) t = relu(t);
    dense(W[2], bb[2], b.data(), F, F, a.data());
    for (double& t : a) t = relu(t);
    if (head == 0) {
      dense(W[3], bb[3], a.data(), A, F, logits);
      if (legal)
        for (int k = 0; k < A; ++k)
          if (!legal[k]) logits[k] = -INFINITY;
    } else {
      dense(W[3], bb[3], a.data(), 1, F, value);
    }
  }
}

extern "C" void orc_s5_step(const orc_s5_net* net, const uint8_t* obs, const uint8_t* reset,
                            const uint8_t* legal, int64_t n, double* state, double* logits,
                            double* values, int32_t n_threads) {
  const int H = net->H, P = net->P, A = net->n_actions;
  auto one = [&](int64_t e) {
    std::vector<double> u(H), y(H), v(H);
    orc_s5_encode(net, obs + e * net->obs_dim, u.data());
    orc_s5_ssm_step(net, u.data(), reset[e], state + e * 2 * P, y.data());
    for (int h = 0; h < H; ++h) v[h] = u[h] + gelu(y[h]);
    orc_s5_heads(net, v.data(), legal ? legal + e * A : nullptr, logits + e * A, values + e);
  };
  const int nt = n_threads > 1 ? n_threads : 1;
  std::vector<std::thread> pool;
  for (int t = 0; t < nt; ++t)
    pool.emplace_back([&, t] {
      for (int64_t e = t; e < n; e += nt) one(e);
    });
  for (auto& th : pool) th.join();
}
