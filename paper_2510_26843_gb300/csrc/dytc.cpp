// Dynamic Tree Cascade (DyTC) scheduling: host code, no GPU work.
//
//   * Sec. 3: expected walltime improvement factors (EWIF) of speculative decoding and of the
//     vertical / horizontal cascades under i.i.d. Bernoulli acceptance;
//   * Sec. 4.2: per-configuration acceptance estimates, alpha <- lambda alpha + (1 - lambda) alpha_recent
//     with alpha_recent the mean of the last H first-draft-token outcomes, updated only for the
//     configurations used in a step (App. D);
//   * Eq. 5 / App. D Algorithm 2: the (configuration, draft length) maximising the local speedup plus
//     the least future speedup of the bottom draft;
//   * Algorithm 1: expand the active leaf of highest accumulated acceptance until the stop rule
//     (alpha_dn / c_dn * P_acc < t_min) or the tree size limit, the drafted tokens coming from the
//     caller (the tree steps of the chosen draft configuration).  With K candidates per drafted
//     position (top-K), the candidates are normalised over the K and kept in rank order while the
//     mass kept before them is below P_tree (top-P, the first always); each child gets
//     P_acc(parent) * alpha(cfg) * its normalised probability (the token-level refinement of
//     Sec. 4.2), and the top-1 child continues the branch.  Expanding a leaf with a neural draft
//     also extends its active siblings in the same draft steps (tree-based parallel drafting).
// An expanded node stops being an active leaf (Algorithm 1 as printed never clears it, which would
// let the same sequence be drafted twice).  Ties keep the first maximum and the lowest node index.
#include <cmath>
#include <cstdint>
#include <cstring>
#include <new>
#include <vector>

#include "../../include/casspec.h"

namespace {

double pow_int(double x, int e) {
  double r = 1.0;
  for (int i = 0; i < e; ++i) r *= x;
  return r;
}

// generating function of the tokens one speculative round of draft length k yields (Sec. 3)
double pgf_round(double a, int k, double x) {
  const double ax = a * x;
  if (std::fabs(1.0 - ax) < 1e-15) return 1.0 + (x - 1.0) * (k + 1);
  return 1.0 + (x - 1.0) * (1.0 - pow_int(ax, k + 1)) / (1.0 - ax);
}

bool bad_alpha(double a) { return !(a >= 0.0 && a <= 1.0); }

}  // namespace

struct casspec_dytc {
  casspec_dytc_params p;
  std::vector<double> alpha, cost;
  std::vector<std::vector<uint8_t>> hist;  // last `window` first-token outcomes per configuration
  std::vector<uint8_t> used;               // recorded since the last end of step
  // draft tree (Algorithm 1)
  std::vector<int32_t> parent, token, cfg;
  std::vector<double> p_acc;
  std::vector<uint8_t> active;
  // measured steps for the latency model, one regression per arithmetic class: bytes moved and
  // microseconds (the most recent kObs of each class)
  std::vector<double> obs_x[CASSPEC_DYTC_MAX_CLASS], obs_y[CASSPEC_DYTC_MAX_CLASS];
};

namespace {
constexpr size_t kObs = 512;
}

extern "C" {

double casspec_ewif_sd(double alpha, double c, int k) {
  if (k < 0 || bad_alpha(alpha)) return NAN;
  const double num = std::fabs(1.0 - alpha) < 1e-12 ? (double)(k + 1) : (1.0 - pow_int(alpha, k + 1)) / (1.0 - alpha);
  return num / (c * k + 1.0);
}

double casspec_ewif_hc(double a1, double c1, int k1, double a2, double c2, int k2) {
  if (k1 < 0 || k2 < 0 || bad_alpha(a1) || bad_alpha(a2) || a1 == 1.0 || a2 == 1.0) return NAN;
  const double first = (1.0 - pow_int(a1, k1 + 1)) / (1.0 - a1);
  const double second = pow_int(a1, k1) * a2 * (1.0 - pow_int(a2, k2)) / (1.0 - a2);
  return (first + second) / (1.0 + k1 * c1 + k2 * c2);
}

double casspec_ewif_vc(double alpha, double alpha12, double c1, double c2, int n, int k) {
  if (n < 0 || k < 0 || bad_alpha(alpha) || bad_alpha(alpha12) || alpha == 1.0) return NAN;
  const double phi = pgf_round(alpha12, k, alpha);
  return (1.0 - alpha * pow_int(phi, n)) / ((1.0 - alpha) * (1.0 + n * c1 + n * k * c2));
}

double casspec_dytc_objective(double alpha, double c, int k, double alpha_dn, double c_dn) {
  if (k < 1 || bad_alpha(alpha)) return NAN;
  const double den = c * k + c_dn;
  if (std::fabs(den) < 1e-12) return NAN;  // Algorithm 2 skips the pair
  const double e_acc = std::fabs(1.0 - alpha) < 1e-9 ? (double)k : alpha * (1.0 - pow_int(alpha, k)) / (1.0 - alpha);
  return (e_acc + pow_int(alpha, k) * alpha_dn) / den;
}

int casspec_dytc_create(const casspec_dytc_params* p, const double* alpha_init, const double* cost, casspec_dytc** out) {
  if (p == nullptr || alpha_init == nullptr || cost == nullptr || out == nullptr) return CASSPEC_E_INVAL;
  if (p->n_cfg < 1 || p->n_cfg > CASSPEC_DYTC_MAX_CFG || p->k_max < 1 || p->k_max > CASSPEC_MAX_TREE || p->m_max < 1 ||
      p->m_max > CASSPEC_MAX_TREE ||
      p->window < 1 || !(p->lambda >= 0.0 && p->lambda <= 1.0) || bad_alpha(p->alpha_dn) || p->c_dn < 0.0 ||
      p->topk < 1 || p->topk > CASSPEC_TOPK_MAX || !(p->p_tree > 0.0 && p->p_tree <= 1.0))
    return CASSPEC_E_INVAL;
  for (int i = 0; i < p->n_cfg; ++i)
    if (bad_alpha(alpha_init[i]) || !(cost[i] >= 0.0)) return CASSPEC_E_INVAL;
  casspec_dytc* s = new (std::nothrow) casspec_dytc;
  if (s == nullptr) return CASSPEC_E_CAPACITY;
  s->p = *p;
  s->alpha.assign(alpha_init, alpha_init + p->n_cfg);
  s->cost.assign(cost, cost + p->n_cfg);
  s->hist.assign(p->n_cfg, {});
  s->used.assign(p->n_cfg, 0);
  *out = s;
  return casspec_dytc_tree_reset(s);
}

void casspec_dytc_destroy(casspec_dytc* s) { delete s; }

int casspec_dytc_get_params(const casspec_dytc* s, casspec_dytc_params* out) {
  if (s == nullptr || out == nullptr) return CASSPEC_E_INVAL;
  *out = s->p;
  return CASSPEC_OK;
}

int casspec_dytc_set_cost(casspec_dytc* s, int cfg, double cost) {
  if (s == nullptr || cfg < 0 || cfg >= s->p.n_cfg || !(cost >= 0.0)) return CASSPEC_E_INVAL;
  s->cost[cfg] = cost;
  return CASSPEC_OK;
}

int casspec_dytc_alpha(const casspec_dytc* s, int cfg, double* alpha_out) {
  if (s == nullptr || alpha_out == nullptr || cfg < 0 || cfg >= s->p.n_cfg) return CASSPEC_E_INVAL;
  *alpha_out = s->alpha[cfg];
  return CASSPEC_OK;
}

int casspec_dytc_cost(const casspec_dytc* s, int cfg, double* cost_out) {
  if (s == nullptr || cost_out == nullptr || cfg < 0 || cfg >= s->p.n_cfg) return CASSPEC_E_INVAL;
  *cost_out = s->cost[cfg];
  return CASSPEC_OK;
}

int casspec_dytc_best_config(const casspec_dytc* s, int* cfg_out, int* k_out, double* obj_out) {
  if (s == nullptr || cfg_out == nullptr || k_out == nullptr) return CASSPEC_E_INVAL;
  double best = -INFINITY;
  int sb = -1, kb = 0;
  for (int c = 0; c < s->p.n_cfg; ++c)
    for (int k = 1; k <= s->p.k_max; ++k) {
      const double v = casspec_dytc_objective(s->alpha[c], s->cost[c], k, s->p.alpha_dn, s->p.c_dn);
      if (std::isnan(v)) continue;
      if (v > best) {
        best = v;
        sb = c;
        kb = k;
      }
    }
  if (!(best > 0.0)) {
    sb = -1;
    kb = 0;
  }
  *cfg_out = sb;
  *k_out = kb;
  if (obj_out) *obj_out = best;
  return CASSPEC_OK;
}

int casspec_dytc_record(casspec_dytc* s, int cfg, int accepted) {
  if (s == nullptr || cfg < 0 || cfg >= s->p.n_cfg) return CASSPEC_E_INVAL;
  auto& h = s->hist[cfg];
  h.push_back(accepted ? 1 : 0);
  if ((int)h.size() > s->p.window) h.erase(h.begin());
  s->used[cfg] = 1;
  return CASSPEC_OK;
}

int casspec_dytc_end_step(casspec_dytc* s) {
  if (s == nullptr) return CASSPEC_E_INVAL;
  for (int c = 0; c < s->p.n_cfg; ++c) {
    if (!s->used[c] || s->hist[c].empty()) continue;
    double sum = 0.0;
    for (uint8_t o : s->hist[c]) sum += o;
    const double recent = sum / (double)s->hist[c].size();
    s->alpha[c] = s->p.lambda * s->alpha[c] + (1.0 - s->p.lambda) * recent;
    s->used[c] = 0;
  }
  return CASSPEC_OK;
}

int casspec_dytc_tree_reset(casspec_dytc* s) {
  if (s == nullptr) return CASSPEC_E_INVAL;
  s->parent.assign(1, -1);
  s->token.assign(1, -1);
  s->cfg.assign(1, -1);
  s->p_acc.assign(1, 1.0);
  s->active.assign(1, 1);
  return CASSPEC_OK;
}

int casspec_dytc_tree_plan(casspec_dytc* s, int* leaf_out, int* cfg_out, int* k_out) {
  if (s == nullptr || leaf_out == nullptr || cfg_out == nullptr || k_out == nullptr) return CASSPEC_E_INVAL;
  *leaf_out = -1;
  *cfg_out = -1;
  *k_out = 0;
  const int n = (int)s->parent.size();
  if (n >= s->p.m_max) return 0;
  int leaf = -1;
  for (int i = 0; i < n; ++i)
    if (s->active[i] && (leaf < 0 || s->p_acc[i] > s->p_acc[leaf])) leaf = i;
  if (leaf < 0) return 0;
  if (s->p.c_dn > 0.0 && s->p.alpha_dn / s->p.c_dn * s->p_acc[leaf] < s->p.t_min) return 0;  // stop rule
  int c = -1, k = 0;
  casspec_dytc_best_config(s, &c, &k, nullptr);
  if (c < 0) {
    s->active[leaf] = 0;
    return 0;
  }
  *leaf_out = leaf;
  *cfg_out = c;
  *k_out = k;
  return 1;
}

int casspec_dytc_tree_extend(casspec_dytc* s, int leaf, int cfg, int k, const int32_t* tokens) {
  if (s == nullptr || tokens == nullptr || cfg < 0 || cfg >= s->p.n_cfg || k < 1) return CASSPEC_E_INVAL;
  const int n0 = (int)s->parent.size();
  if (leaf < 0 || leaf >= n0 || !s->active[leaf]) return CASSPEC_E_INVAL;
  s->active[leaf] = 0;
  int node = leaf, added = 0;
  for (int i = 0; i < k && (int)s->parent.size() < s->p.m_max; ++i) {
    s->parent.push_back(node);
    s->token.push_back(tokens[i]);
    s->cfg.push_back(cfg);
    s->p_acc.push_back(s->p_acc[node] * s->alpha[cfg]);
    s->active.push_back(1);
    if (node != leaf) s->active[node] = 0;
    node = (int)s->parent.size() - 1;
    ++added;
  }
  return added;
}

int casspec_dytc_tree_begin(casspec_dytc* s, int leaf, int siblings, int32_t* branches_out, int* nb_out) {
  if (s == nullptr || branches_out == nullptr || nb_out == nullptr) return CASSPEC_E_INVAL;
  const int n = (int)s->parent.size();
  if (leaf < 0 || leaf >= n || !s->active[leaf]) return CASSPEC_E_INVAL;
  int nb = 0;
  branches_out[nb++] = leaf;
  if (siblings && leaf != 0)
    for (int j = 0; j < n; ++j)
      if (j != leaf && s->active[j] && s->parent[j] == s->parent[leaf]) branches_out[nb++] = j;
  *nb_out = nb;
  return CASSPEC_OK;
}

int casspec_dytc_tree_add(casspec_dytc* s, int node, int cfg, const int32_t* tokens, const float* probs, int kc) {
  if (s == nullptr || tokens == nullptr || probs == nullptr || cfg < 0 || cfg >= s->p.n_cfg || kc < 1 ||
      kc > CASSPEC_TOPK_MAX)
    return CASSPEC_E_INVAL;
  const int n0 = (int)s->parent.size();
  if (node < 0 || node >= n0) return CASSPEC_E_INVAL;
  if (n0 >= s->p.m_max) return 0;
  double total = 0.0;
  for (int j = 0; j < kc; ++j) {
    if (!(probs[j] >= 0.0f)) return CASSPEC_E_INVAL;
    total += (double)probs[j];
  }
  if (!(total > 0.0)) return CASSPEC_E_INVAL;
  s->active[node] = 0;  // it receives children
  const double base = s->p_acc[node] * s->alpha[cfg];
  double mass = 0.0;
  for (int j = 0; j < kc && (int)s->parent.size() < s->p.m_max; ++j) {
    if (j > 0 && mass >= s->p.p_tree) break;
    const double q = (double)probs[j] / total;
    s->parent.push_back(node);
    s->token.push_back(tokens[j]);
    s->cfg.push_back(cfg);
    s->p_acc.push_back(base * q);
    s->active.push_back(1);
    mass += q;
  }
  return n0;  // the top-1 child
}

int casspec_vc_accept(const int32_t* proposals, int j, const int32_t* argmax, int32_t* out) {
  if (j < 0 || (j > 0 && proposals == nullptr) || argmax == nullptr || out == nullptr) return CASSPEC_E_INVAL;
  int a = 0;
  while (a < j && proposals[a] == argmax[a]) {
    out[a] = proposals[a];
    ++a;
  }
  out[a] = argmax[a];  // d_i's own next token after the accepted prefix
  return a + 1;
}

int casspec_dytc_tree_get(const casspec_dytc* s, int* n_out, int32_t* parent_out, int32_t* token_out, int32_t* cfg_out,
                          double* p_acc_out) {
  if (s == nullptr || n_out == nullptr) return CASSPEC_E_INVAL;
  const int n = (int)s->parent.size();
  *n_out = n;
  if (parent_out) std::memcpy(parent_out, s->parent.data(), n * sizeof(int32_t));
  if (token_out) std::memcpy(token_out, s->token.data(), n * sizeof(int32_t));
  if (cfg_out) std::memcpy(cfg_out, s->cfg.data(), n * sizeof(int32_t));
  if (p_acc_out) std::memcpy(p_acc_out, s->p_acc.data(), n * sizeof(double));
  return CASSPEC_OK;
}

double casspec_step_bytes(const casspec_model_config* c, const uint8_t* skip_mask, int quant_mode, int n, int P) {
  if (c == nullptr || c->n_layers < 1 || c->d_model < 1 || c->ffn < 1 || c->vocab < 1 || n < 0 || P < 0 ||
      quant_mode < 0 || quant_mode > 2)
    return -1.0;
  const double d = c->d_model, F = c->ffn, V = c->vocab;
  const double wb = quant_mode == 2 ? 0.5 : (quant_mode == 1 ? 1.0 : 2.0);  // bytes per weight
  const double sb = quant_mode != 0 ? 4.0 : 0.0;                            // bytes per row scale
  double bytes = V * d * 2.0 + (double)n * V * 4.0;  // LM head read, fp32 logits written
  for (int l = 0; l < c->n_layers; ++l) {
    const uint8_t code = skip_mask ? skip_mask[l] : 1;
    if (code == 0) continue;
    if (!(code & CASSPEC_SKIP_ATTN))  // Wqkv, Wo (+ scales), the prefix K/V read, the new K/V written
      bytes += 4.0 * d * d * wb + 4.0 * d * sb + 2.0 * P * d * 2.0 + 2.0 * n * d * 2.0;
    if (!(code & CASSPEC_SKIP_FFN))  // Wg, Wu, Wd (+ scales)
      bytes += 3.0 * d * F * wb + (2.0 * F + d) * sb;
  }
  return bytes;
}

int casspec_dytc_observe(casspec_dytc* s, int cls, double bytes, double us) {
  if (s == nullptr || cls < 0 || cls >= CASSPEC_DYTC_MAX_CLASS || !(bytes >= 0.0) || !(us > 0.0))
    return CASSPEC_E_INVAL;
  std::vector<double>& x = s->obs_x[cls];
  std::vector<double>& y = s->obs_y[cls];
  if (x.size() == kObs) {
    x.erase(x.begin());
    y.erase(y.begin());
  }
  x.push_back(bytes);
  y.push_back(us);
  return CASSPEC_OK;
}

int casspec_dytc_fit_costs(casspec_dytc* s, const int* cfg_class, const double* cfg_bytes, double target_bytes,
                           const double* mu0, const double* sd0, double noise_sd, double* w_out) {
  if (s == nullptr || cfg_class == nullptr || cfg_bytes == nullptr || !(target_bytes > 0.0)) return CASSPEC_E_INVAL;
  for (int c = 0; c < s->p.n_cfg; ++c)
    if (!(cfg_bytes[c] >= 0.0) || cfg_class[c] < 0 || cfg_class[c] >= CASSPEC_DYTC_MAX_CLASS) return CASSPEC_E_INVAL;
  // one posterior per class (a class without measured steps keeps the prior)
  double w[CASSPEC_DYTC_MAX_CLASS][2];
  for (int k = 0; k < CASSPEC_DYTC_MAX_CLASS; ++k) {
    const int m = (int)s->obs_x[k].size();
    const int rc = casspec_latency_fit(m ? s->obs_x[k].data() : nullptr, m ? s->obs_y[k].data() : nullptr, m, mu0,
                                       sd0, noise_sd, w[k], nullptr);
    if (rc != CASSPEC_OK) return rc;
  }
  const double t_target = w[0][0] + w[0][1] * target_bytes;
  if (!(t_target > 0.0)) return CASSPEC_E_INVAL;
  for (int c = 0; c < s->p.n_cfg; ++c) {
    const double* wc = w[cfg_class[c]];
    s->cost[c] = std::fmax(wc[0] + wc[1] * cfg_bytes[c], 0.0) / t_target;
  }
  if (w_out)
    for (int k = 0; k < CASSPEC_DYTC_MAX_CLASS; ++k) {
      w_out[2 * k] = w[k][0];
      w_out[2 * k + 1] = w[k][1];
    }
  return CASSPEC_OK;
}

int casspec_latency_fit(const double* x, const double* y, int m, const double* mu0, const double* sd0, double noise_sd,
                        double* w_out, double* cov_out) {
  if ((m > 0 && (x == nullptr || y == nullptr)) || m < 0 || mu0 == nullptr || sd0 == nullptr || w_out == nullptr ||
      !(sd0[0] > 0.0) || !(sd0[1] > 0.0) || !(noise_sd > 0.0))
    return CASSPEC_E_INVAL;
  // Solved in the scaled regressor u = x / xs (w1 scaled to w1 xs with its prior) so that the 2 x 2
  // system stays well conditioned whatever unit x comes in; precision = S0^-1 + U^T U / s^2,
  // rhs = S0^-1 mu0 + U^T y / s^2.
  double xs = 0.0;
  for (int i = 0; i < m; ++i) xs = std::fmax(xs, std::fabs(x[i]));
  if (!(xs > 0.0)) xs = 1.0;
  const double is2 = 1.0 / (noise_sd * noise_sd);
  const double sd1 = sd0[1] * xs, mu1 = mu0[1] * xs;
  double a = 1.0 / (sd0[0] * sd0[0]), b = 0.0, d = 1.0 / (sd1 * sd1);
  double r0 = mu0[0] * a, r1 = mu1 * d;
  for (int i = 0; i < m; ++i) {
    const double u = x[i] / xs;
    a += is2;
    b += u * is2;
    d += u * u * is2;
    r0 += y[i] * is2;
    r1 += u * y[i] * is2;
  }
  const double det = a * d - b * b;
  if (!(det > 0.0)) return CASSPEC_E_INVAL;
  const double c00 = d / det, c01 = -b / det, c11 = a / det;
  w_out[0] = c00 * r0 + c01 * r1;
  w_out[1] = (c01 * r0 + c11 * r1) / xs;
  if (cov_out) {
    cov_out[0] = c00;
    cov_out[1] = c01 / xs;
    cov_out[2] = c01 / xs;
    cov_out[3] = c11 / (xs * xs);
  }
  return CASSPEC_OK;
}

}  // extern "C"
