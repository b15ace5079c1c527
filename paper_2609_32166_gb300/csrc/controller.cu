// Proposal-length controller (Section 3.2, eq. 1): host code, no GPU.
//
// Runs once per decoding iteration between verify steps, so it is plain
// double-precision C with no allocation: the argmin over l <= l_max of the
// estimated iteration latency per produced token, with the two logistic
// acceptance estimators and the log-quadratic latency estimator updated
// from each iteration's outcome.  The arithmetic follows the order of the
// definitions (sums left to right, no fused multiply-adds: host code is
// built with -ffp-contract=off) so that results are reproducible.
#include <cmath>
#include <cstdio>

#include "pf_internal.h"

namespace {

double sigmoid(double z) { return 1.0 / (1.0 + std::exp(-z)); }

double dot3(const double* w, const double* x) {
  double s = 0.0;
  for (int i = 0; i < 3; ++i) s += w[i] * x[i];
  return s;
}

void logistic_step(double* w, const double* x, double y, double lr) {
  const double g = y - sigmoid(dot3(w, x));
  for (int i = 0; i < 3; ++i) w[i] += lr * g * x[i];
}

// A(l) = sum_{k=1..l} p1 pc^(k-1)
double expected_accepted(double p1, double pc, int ell) {
  double a = 0.0;
  for (int k = 1; k <= ell; ++k) a += p1 * std::pow(pc, (double)(k - 1));
  return a;
}

void latency_features(const pf_length_controller* c, int ell, double* x) {
  const double u = (double)ell / (double)c->l_max;
  x[0] = 1.0;
  x[1] = u;
  x[2] = u * u;
}

double predict_latency(const pf_length_controller* c, int ell) {
  double x[3];
  latency_features(c, ell, x);
  return std::exp(c->c[0] * x[0] + c->c[1] * x[1] + c->c[2] * x[2]);
}

void predict_accept(const pf_length_controller* c, int ell, double s, double* p1, double* pc) {
  const double x[3] = {1.0, (double)ell / (double)c->l_max, s};
  *p1 = sigmoid(dot3(c->w_first, x));
  *pc = sigmoid(dot3(c->w_cont, x));
}

}  // namespace

extern "C" {

pf_status pf_length_select(const double* t_hat, const double* p_first, const double* p_cont,
                           int32_t l_max, int32_t* ell_out, double* objective_out) {
  static const char* who = "pf_length_select";
  if (!t_hat || !p_first || !p_cont || !ell_out)
    return pf::set_error(PF_ERR_NULL, "%s: a required pointer is NULL", who);
  if (l_max < 0 || l_max > PF_CTL_MAX_LEN)
    return pf::set_error(PF_ERR_SHAPE, "%s: l_max must be in [0, %d]", who, PF_CTL_MAX_LEN);
  int best = 0;
  double best_obj = 0.0;
  for (int ell = 0; ell <= l_max; ++ell) {
    const double obj = t_hat[ell] / (expected_accepted(p_first[ell], p_cont[ell], ell) + 1.0);
    if (ell == 0 || obj < best_obj) {
      best = ell;
      best_obj = obj;
    }
  }
  *ell_out = best;
  if (objective_out) *objective_out = best_obj;
  return PF_OK;
}

pf_status pf_controller_init(pf_length_controller* c, int32_t l_max, double lr, double epsilon) {
  static const char* who = "pf_controller_init";
  if (!c) return pf::set_error(PF_ERR_NULL, "%s: controller is NULL", who);
  if (l_max < 1 || l_max > PF_CTL_MAX_LEN || !(lr > 0.0) || !(epsilon >= 0.0 && epsilon <= 1.0))
    return pf::set_error(PF_ERR_SHAPE, "%s: need 1 <= l_max <= %d, lr > 0, 0 <= epsilon <= 1",
                         who, PF_CTL_MAX_LEN);
  *c = pf_length_controller{};
  c->l_max = l_max;
  c->lr = lr;
  c->epsilon = epsilon;
  for (int i = 0; i < 3; ++i) c->P[i * 3 + i] = 1e8;
  return PF_OK;
}

pf_status pf_controller_observe(pf_length_controller* c, int32_t ell, double similarity,
                                int32_t accepted, double latency_us) {
  static const char* who = "pf_controller_observe";
  if (!c) return pf::set_error(PF_ERR_NULL, "%s: controller is NULL", who);
  if (ell < 0 || ell > c->l_max || accepted > ell)
    return pf::set_error(PF_ERR_SHAPE, "%s: need 0 <= ell <= l_max and accepted <= ell", who);
  if (accepted >= 0 && ell >= 1) {
    const double x[3] = {1.0, (double)ell / (double)c->l_max, similarity};
    logistic_step(c->w_first, x, accepted >= 1 ? 1.0 : 0.0, c->lr);
    if (accepted >= 1) {
      const int last = accepted + 1 < ell ? accepted + 1 : ell;
      for (int k = 2; k <= last; ++k) logistic_step(c->w_cont, x, k <= accepted ? 1.0 : 0.0, c->lr);
    }
  }
  if (latency_us > 0.0) {
    double x[3];
    latency_features(c, ell, x);
    const double y = std::log(latency_us);
    double Px[3];
    for (int i = 0; i < 3; ++i) Px[i] = dot3(c->P + 3 * i, x);
    double xPx = 0.0;
    for (int i = 0; i < 3; ++i) xPx += x[i] * Px[i];
    const double denom = 1.0 + xPx;
    double k[3];
    for (int i = 0; i < 3; ++i) k[i] = Px[i] / denom;
    const double err = y - dot3(c->c, x);
    for (int i = 0; i < 3; ++i) c->c[i] = c->c[i] + k[i] * err;
    for (int i = 0; i < 3; ++i)
      for (int j = 0; j < 3; ++j) c->P[i * 3 + j] = c->P[i * 3 + j] - k[i] * Px[j];
    c->n_latency += 1;
  }
  return PF_OK;
}

pf_status pf_controller_choose(const pf_length_controller* c, double similarity, double u,
                               double u_dir, int32_t* ell_out, double* objective_out) {
  static const char* who = "pf_controller_choose";
  if (!c || !ell_out) return pf::set_error(PF_ERR_NULL, "%s: a required pointer is NULL", who);
  int best = 0;
  double best_obj = 0.0;
  for (int ell = 0; ell <= c->l_max; ++ell) {
    double p1, pc;
    predict_accept(c, ell, similarity, &p1, &pc);
    const double obj = predict_latency(c, ell) / (expected_accepted(p1, pc, ell) + 1.0);
    if (ell == 0 || obj < best_obj) {
      best = ell;
      best_obj = obj;
    }
  }
  if (u < c->epsilon && c->l_max > 0) {
    if (best == 0 || (best < c->l_max && u_dir < 0.5))
      best += 1;
    else
      best -= 1;
  }
  *ell_out = best;
  if (objective_out) *objective_out = best_obj;
  return PF_OK;
}

}  // extern "C"
