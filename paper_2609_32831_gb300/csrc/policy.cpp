// Host policy of UniCache (tens of numbers per layer chunk; no device work).
//
//  uc_concentration       App. B: share of within-type mass on the top 10 %
//  uc_calibrate_policy    §3.2 / App. B: evict if mean concentration >= 0.5
//  uc_allocate_budget     §3.3 Eq. 2 + redistribution, then §3.4's mapping of
//                         a budget to (kept tokens, bit width)
//  uc_retention_schedule  §3.3 Eq. 3
//  uc_retention_step      Eq. 3 with M^(c) formed from a chunk's type masses
//  uc_plan_batch          one segment configuration per (layer, type) for a
//                         batch of per-sequence budgets
//  uc_keep_count          tokens a fixed keep fraction retains
#include <algorithm>
#include <cmath>
#include <cstring>
#include <functional>
#include <vector>

#include "internal.h"

namespace {

constexpr double kBf16TokenBytes = 4.0 * UC_HEAD_DIM;  // K + V, bf16

// Bytes per kept token and KV head for K + V at `bits` in the packed layout:
// codes, V per-token (scale, zero) pairs and K per-channel pairs amortised
// over a group of 32 tokens.
double token_bytes(int bits) {
  if (bits == 16) return kBf16TokenBytes;
  const double codes = 2.0 * UC_HEAD_DIM * bits / 8.0;
  const double v_params = (UC_HEAD_DIM / UC_GROUP) * 4.0;
  const double k_params = UC_HEAD_DIM * 4.0 / UC_GROUP;
  return codes + v_params + k_params;
}

int64_t ceil_frac(int64_t n, double frac) {
  return (int64_t)std::ceil(frac * (double)n - 1e-9);
}

}  // namespace

extern "C" {

uc_status uc_concentration(const float* mass, int64_t n, double top_frac, double* out) {
  UC_TRACE();
  if (mass == nullptr || out == nullptr || n <= 0 || !(top_frac > 0.0) || top_frac > 1.0) {
    uc::set_error("uc_concentration: bad arguments");
    return UC_ERR_ARG;
  }
  std::vector<double> v(mass, mass + n);
  double total = 0.0;
  for (double x : v) {
    if (!std::isfinite(x) || x < 0.0) {
      uc::set_error("uc_concentration: mass must be finite and non-negative");
      return UC_ERR_RANGE;
    }
    total += x;
  }
  if (total <= 0.0) {
    *out = 0.0;
    return UC_OK;
  }
  const int64_t k = std::max<int64_t>(1, ceil_frac(n, top_frac));
  std::nth_element(v.begin(), v.begin() + (k - 1), v.end(), std::greater<double>());
  double top = 0.0;
  for (int64_t i = 0; i < k; ++i) top += v[i];
  *out = top / total;
  return UC_OK;
}

uc_status uc_calibrate_policy(uc_segment_table* t, const float* const* mass, int32_t n_examples,
                              double top_frac, double threshold) {
  UC_TRACE();
  if (t == nullptr || mass == nullptr || n_examples <= 0 || t->n_types <= 0 ||
      t->n_types > UC_MAX_SEGMENTS) {
    uc::set_error("uc_calibrate_policy: bad arguments");
    return UC_ERR_ARG;
  }
  for (int a = 0; a < t->n_types; ++a) {
    if (!t->candidate[a]) {
      t->policy[a] = UC_POLICY_PROTECTED;
      t->concentration[a] = 0.0;
      continue;
    }
    double sum = 0.0;
    for (int e = 0; e < n_examples; ++e) {
      const float* m = mass[(size_t)e * t->n_types + a];
      double c = 0.0;
      const uc_status st = uc_concentration(m, t->n_tokens[a], top_frac, &c);
      if (st != UC_OK) return st;
      sum += c;
    }
    t->concentration[a] = sum / n_examples;
    t->policy[a] = (t->concentration[a] >= threshold) ? UC_POLICY_EVICT : UC_POLICY_QUANT;
  }
  return UC_OK;
}

uc_status uc_allocate_budget(uc_segment_table* t, double rho, int32_t first_chunk) {
  UC_TRACE();
  if (t == nullptr || t->n_types <= 0 || t->n_types > UC_MAX_SEGMENTS || !(rho >= 0.0) || rho > 1.0) {
    uc::set_error("uc_allocate_budget: bad arguments (need 0 <= rho <= 1)");
    return UC_ERR_ARG;
  }
  const int n = t->n_types;
  double m[UC_MAX_SEGMENTS], cap[UC_MAX_SEGMENTS], b[UC_MAX_SEGMENTS];
  double msum = 0.0, total = 0.0;
  for (int a = 0; a < n; ++a)
    if (t->candidate[a]) total += kBf16TokenBytes * t->n_tokens[a];
  total *= rho;
  for (int a = 0; a < n; ++a) {
    m[a] = t->candidate[a] ? t->mass[a] : 0.0;
    cap[a] = first_chunk ? kBf16TokenBytes * t->n_tokens[a] : t->budget[a];
    if (t->candidate[a] && (!(m[a] >= 0.0) || !std::isfinite(m[a]) || !(cap[a] >= 0.0))) {
      uc::set_error("uc_allocate_budget: mass and budgets must be finite and non-negative");
      return UC_ERR_RANGE;
    }
    b[a] = 0.0;
    msum += m[a];
  }
  // Eq. 2: proportional share of the shared budget, capped by the previous
  // allocation; leftovers go to uncapped types with positive mass.
  if (msum > 0.0 && total > 0.0) {
    for (int a = 0; a < n; ++a)
      if (t->candidate[a]) b[a] = std::min(cap[a], m[a] / msum * total);
    for (int round = 0; round <= n; ++round) {
      double used = 0.0, open_mass = 0.0;
      for (int a = 0; a < n; ++a) used += b[a];
      for (int a = 0; a < n; ++a)
        if (t->candidate[a] && b[a] < cap[a] && m[a] > 0.0) open_mass += m[a];
      const double rest = total - used;
      if (rest <= 1e-12 * std::max(total, 1.0) || open_mass <= 0.0) break;
      for (int a = 0; a < n; ++a)
        if (t->candidate[a] && b[a] < cap[a] && m[a] > 0.0)
          b[a] = std::min(cap[a], b[a] + rest * m[a] / open_mass);
    }
  }
  // §3.4: budget -> policy configuration
  for (int a = 0; a < n; ++a) {
    const int64_t ntok = t->n_tokens[a];
    if (!t->candidate[a]) {
      t->kind[a] = UC_KIND_FULL;
      t->keep[a] = (int32_t)ntok;
      t->bits[a] = 16;
      continue;
    }
    t->budget[a] = b[a];
    if (ntok <= 0) {
      t->keep[a] = 0;
      t->bits[a] = 16;
      t->kind[a] = UC_KIND_EVICT;
      continue;
    }
    if (t->policy[a] == UC_POLICY_EVICT) {
      int64_t keep = (int64_t)std::floor(b[a] / token_bytes(16) + 1e-9);
      keep = std::max<int64_t>(1, std::min(ntok, keep));
      t->keep[a] = (int32_t)keep;
      t->bits[a] = 16;
      t->kind[a] = keep == ntok ? UC_KIND_FULL : UC_KIND_EVICT;
    } else if (t->policy[a] == UC_POLICY_QUANT) {
      int bits = 0;
      for (int cand : {4, 2})
        if ((double)ntok * token_bytes(cand) <= b[a] * (1.0 + 1e-12)) {
          bits = cand;
          break;
        }
      if (bits) {
        t->keep[a] = (int32_t)ntok;
        t->bits[a] = bits;
        t->kind[a] = UC_KIND_QUANT;
      } else {
        int64_t keep = (int64_t)std::floor(b[a] / token_bytes(2) + 1e-9);
        keep = std::max<int64_t>(1, std::min(ntok, keep));
        t->keep[a] = (int32_t)keep;
        t->bits[a] = 2;
        t->kind[a] = UC_KIND_EVICT_QUANT;
      }
    } else {
      uc::set_error("uc_allocate_budget: candidate type %d has no policy", a);
      return UC_ERR_ARG;
    }
  }
  return UC_OK;
}

uc_status uc_retention_schedule(double rho_prev, double rho_init, double rho_min, double m_c,
                                double m_0, double* rho_out) {
  UC_TRACE();
  if (rho_out == nullptr || !(rho_min > 0.0) || rho_min > rho_init || rho_init > 1.0 ||
      !(m_0 > 0.0) || !(m_c >= 0.0)) {
    uc::set_error("uc_retention_schedule: need 0 < rho_min <= rho_init <= 1, M0 > 0, M >= 0");
    return UC_ERR_ARG;
  }
  *rho_out = std::min(rho_prev, std::max(rho_min, rho_init * m_c / m_0));
  return UC_OK;
}

uc_status uc_keep_count(int32_t n, double keep_frac, int32_t* out) {
  UC_TRACE();
  if (out == nullptr || !(keep_frac > 0.0) || keep_frac > 1.0 || n < 0) {
    uc::set_error("uc_keep_count: need 0 < keep_frac <= 1 and n >= 0");
    return UC_ERR_ARG;
  }
  if (n == 0) {
    *out = 0;
    return UC_OK;
  }
  const int64_t k = (int64_t)std::floor(keep_frac * (double)n + 1e-9);
  *out = (int32_t)std::max<int64_t>(1, std::min<int64_t>(n, k));
  return UC_OK;
}

uc_status uc_plan_batch(const uc_segment_table* tables, int32_t n_seq, int32_t type, int32_t* keep,
                        uc_type_config* out) {
  UC_TRACE();
  if (tables == nullptr || keep == nullptr || out == nullptr || n_seq < 1 || tables[0].n_types < 1 ||
      tables[0].n_types > UC_MAX_SEGMENTS || type < 0 || type >= tables[0].n_types) {
    uc::set_error("uc_plan_batch: bad arguments");
    return UC_ERR_ARG;
  }
  const int n = tables[0].n_tokens[type];
  bool all_full = true, all_tokens = true;
  int bits = 16, max_keep = 0;
  for (int b = 0; b < n_seq; ++b) {
    const uc_segment_table& t = tables[b];
    if (t.n_types != tables[0].n_types || t.n_tokens[type] != n || t.candidate[type] != tables[0].candidate[type]) {
      uc::set_error("uc_plan_batch: the sequences' tables describe different types");
      return UC_ERR_SHAPE;
    }
    const int k = t.candidate[type] ? t.keep[type] : n;
    if (k < 0 || k > n || (t.candidate[type] && t.bits[type] != 16 && t.bits[type] != 4 && t.bits[type] != 2)) {
      uc::set_error("uc_plan_batch: table %d has no configuration for type %d (uc_allocate_budget first)", b, type);
      return UC_ERR_ARG;
    }
    keep[b] = k;
    max_keep = std::max(max_keep, k);
    all_tokens &= k == n;
    if (t.candidate[type]) {
      all_full &= t.kind[type] == UC_KIND_FULL;
      bits = std::min(bits, (int)t.bits[type]);
    }
  }
  out->max_keep = max_keep;
  if (all_full) {  // every sequence keeps every token in bf16: a view of the rows
    out->kind = UC_KIND_FULL;
    out->bits = 16;
    out->full_view = 1;
    return UC_OK;
  }
  out->full_view = 0;
  out->bits = bits;
  out->kind = bits == 16 ? UC_KIND_EVICT : (all_tokens ? UC_KIND_QUANT : UC_KIND_EVICT_QUANT);
  return UC_OK;
}

uc_status uc_retention_step(const uc_segment_table* t, int32_t first_chunk, double rho_prev, double rho_init,
                            double rho_min, double* m_0, double* rho_out) {
  UC_TRACE();
  if (t == nullptr || m_0 == nullptr || rho_out == nullptr || t->n_types < 1 || t->n_types > UC_MAX_SEGMENTS) {
    uc::set_error("uc_retention_step: bad arguments");
    return UC_ERR_ARG;
  }
  double m_c = 0.0;  // M^(c): the mass on every candidate type
  for (int a = 0; a < t->n_types; ++a)
    if (t->candidate[a]) {
      if (!(t->mass[a] >= 0.0) || !std::isfinite(t->mass[a])) {
        uc::set_error("uc_retention_step: masses must be finite and non-negative");
        return UC_ERR_RANGE;
      }
      m_c += t->mass[a];
    }
  if (first_chunk) {
    if (!(rho_min > 0.0) || rho_min > rho_init || rho_init > 1.0) {
      uc::set_error("uc_retention_step: need 0 < rho_min <= rho_init <= 1");
      return UC_ERR_ARG;
    }
    *m_0 = m_c;
    *rho_out = rho_init;
    return UC_OK;
  }
  if (!(*m_0 > 0.0)) {  // no attention on the candidates at chunk 0: the ratio stays
    *rho_out = rho_prev;
    return UC_OK;
  }
  return uc_retention_schedule(rho_prev, rho_init, rho_min, m_c, *m_0, rho_out);
}

}  // extern "C"
