// Head-level KV budget allocation: Section 3.3 (Eq. 2) and Appendix A.1 (Algorithm 1).
//
// Host-only and deterministic.  Every floating-point step is an IEEE double operation in
// a fixed order; this file must be compiled with -ffp-contract=off so no multiply-add is
// fused, which keeps the integer budgets identical on every machine.
#include <algorithm>
#include <cmath>
#include <cstdint>
#include <vector>

#include "sgdkv.h"

namespace {

// S_h = s_h / sum(s), summed in ascending head order; all-zero scores give uniform shares.
std::vector<double> normalise(const std::vector<double>& s) {
  const size_t n = s.size();
  double total = 0.0;
  for (size_t h = 0; h < n; ++h) total += s[h];
  std::vector<double> S(n);
  for (size_t h = 0; h < n; ++h) S[h] = (total == 0.0) ? 1.0 / double(n) : s[h] / total;
  return S;
}

// Algorithm 1, steps 2-5: cap at M, collect the excess E, walk the uncapped heads by
// descending S_h (lower index first on ties) and fill each up to M until E is spent.
std::vector<double> greedy_redistribute(const std::vector<double>& S,
                                        const std::vector<double>& x, double cap) {
  const int n = int(x.size());
  double excess = 0.0;
  for (int h = 0; h < n; ++h)
    if (x[h] > cap) excess += x[h] - cap;
  std::vector<double> xt(n);
  std::vector<int> order;
  for (int h = 0; h < n; ++h) {
    xt[h] = std::min(x[h], cap);
    if (!(x[h] > cap)) order.push_back(h);
  }
  std::sort(order.begin(), order.end(), [&](int a, int b) {
    if (S[a] != S[b]) return S[a] > S[b];
    return a < b;
  });
  for (int h : order) {
    if (excess <= 0.0) break;
    const double give = std::min(excess, cap - xt[h]);
    xt[h] += give;
    excess -= give;
  }
  return xt;
}

// Water level: x_h = min(cap, lambda * S_h) with sum x_h = pool; heads whose share would
// exceed the cap are pinned there and lambda is re-solved until no new head overflows.
std::vector<double> proportional_waterfill(const std::vector<double>& S, double pool,
                                           double cap) {
  const int n = int(S.size());
  std::vector<char> capped(n, 0);
  int ncapped = 0;
  for (;;) {
    const double free_pool = pool - cap * double(ncapped);
    double ssum = 0.0;
    for (int h = 0; h < n; ++h)
      if (!capped[h]) ssum += S[h];
    std::vector<double> out(n);
    if (ssum <= 0.0) {
      const int rest = n - ncapped;
      for (int h = 0; h < n; ++h)
        out[h] = capped[h] ? cap : (rest > 0 ? free_pool / double(rest) : 0.0);
      return out;
    }
    const double lam = free_pool / ssum;
    int newly = 0;
    for (int h = 0; h < n; ++h)
      if (!capped[h] && lam * S[h] > cap) ++newly;
    if (newly == 0) {
      for (int h = 0; h < n; ++h) out[h] = capped[h] ? cap : lam * S[h];
      return out;
    }
    for (int h = 0; h < n; ++h)
      if (!capped[h] && lam * S[h] > cap) {
        capped[h] = 1;
        ++ncapped;
      }
  }
}

// Largest remainder: floors, then one token at a time to heads ordered by (fractional
// part desc, S_h desc, index asc), skipping heads already at the cap.
bool largest_remainder(const std::vector<double>& S, const std::vector<double>& xt,
                       int64_t pool, int64_t cap, std::vector<int64_t>& m) {
  const int n = int(xt.size());
  m.assign(n, 0);
  std::vector<double> frac(n);
  int64_t assigned = 0;
  for (int h = 0; h < n; ++h) {
    const double fl = std::floor(xt[h]);
    int64_t v = int64_t(fl);
    v = std::min(std::max(v, int64_t(0)), cap);
    m[h] = v;
    assigned += v;
    frac[h] = xt[h] - fl;
  }
  int64_t rest = pool - assigned;
  std::vector<int> order(n);
  for (int h = 0; h < n; ++h) order[h] = h;
  std::sort(order.begin(), order.end(), [&](int a, int b) {
    if (frac[a] != frac[b]) return frac[a] > frac[b];
    if (S[a] != S[b]) return S[a] > S[b];
    return a < b;
  });
  while (rest > 0) {
    bool progressed = false;
    for (int h : order) {
      if (rest == 0) break;
      if (m[h] < cap) {
        ++m[h];
        --rest;
        progressed = true;
      }
    }
    if (!progressed) return false;
  }
  return true;
}

}  // namespace

extern "C" sgdkv_status sgdkv_allocate_budgets(const float* head_scores, int32_t n_heads,
                                               int64_t context_len, int64_t total_budget,
                                               int64_t floor, int32_t mode,
                                               int64_t* budgets_out) {
  if (!head_scores || !budgets_out || n_heads <= 0) return SGDKV_ERR_INVALID_ARG;
  if (context_len <= 0 || context_len > (int64_t(1) << 40)) return SGDKV_ERR_INVALID_ARG;
  if (floor < 0 || floor > context_len) return SGDKV_ERR_INVALID_ARG;
  if (mode < SGDKV_ALLOC_GREEDY || mode > SGDKV_ALLOC_REVERSE) return SGDKV_ERR_INVALID_ARG;
  const int n = n_heads;
  std::vector<double> s(n);
  for (int h = 0; h < n; ++h) {
    const float v = head_scores[h];
    if (!std::isfinite(v) || v < 0.0f) return SGDKV_ERR_INVALID_ARG;
    s[h] = double(v);
  }
  const int64_t C = context_len, f = floor, T = total_budget;
  if (T < int64_t(n) * f || T > int64_t(n) * C) return SGDKV_ERR_INFEASIBLE_BUDGET;

  if (mode == SGDKV_ALLOC_THRESHOLD) {
    double mean = 0.0;
    for (int h = 0; h < n; ++h) mean += s[h];
    mean = mean / double(n);
    for (int h = 0; h < n; ++h)
      if (!(s[h] >= mean)) s[h] = 0.0;
  }
  const std::vector<double> S = normalise(s);
  const int64_t cap = C - f;
  const int64_t pool = T - int64_t(n) * f;
  std::vector<double> x(n);
  for (int h = 0; h < n; ++h) x[h] = S[h] * double(pool);

  std::vector<double> xt = (mode == SGDKV_ALLOC_PROPORTIONAL)
                               ? proportional_waterfill(S, double(pool), double(cap))
                               : greedy_redistribute(S, x, double(cap));
  std::vector<int64_t> m;
  if (!largest_remainder(S, xt, pool, cap, m)) return SGDKV_ERR_INFEASIBLE_BUDGET;
  for (int h = 0; h < n; ++h)
    budgets_out[h] = f + (mode == SGDKV_ALLOC_REVERSE ? cap - m[h] : m[h]);
  return SGDKV_OK;
}

// SGD-KV + HeadKV scores: the mean of the two normalised score sets.
extern "C" sgdkv_status sgdkv_mix_head_scores(const float* a, const float* b, int32_t n_heads,
                                              float* scores_out) {
  if (!a || !b || !scores_out || n_heads <= 0) return SGDKV_ERR_INVALID_ARG;
  const int n = n_heads;
  std::vector<double> sa(n), sb(n);
  for (int h = 0; h < n; ++h) {
    if (!std::isfinite(a[h]) || a[h] < 0.0f || !std::isfinite(b[h]) || b[h] < 0.0f)
      return SGDKV_ERR_INVALID_ARG;
    sa[h] = double(a[h]);
    sb[h] = double(b[h]);
  }
  const std::vector<double> A = normalise(sa), B = normalise(sb);
  for (int h = 0; h < n; ++h) scores_out[h] = float((A[h] + B[h]) / 2.0);
  return SGDKV_OK;
}
