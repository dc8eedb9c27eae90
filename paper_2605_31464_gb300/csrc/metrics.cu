// Host-side evaluation of 8-bin forecasts against measured speedups (no device work).
//
// Bins and representatives follow Table tab:speedup-bins: bin 1 S <= 0.25, 2 (0.25, 0.5],
// 3 (0.5, 0.71], 4 (0.71, 1], 5 (1, 1.41], 6 (1.41, 2], 7 (2, 4], 8 S > 4, upper edges inclusive.
// The scores are those of Sec. 3.1 (speedup recovered over the budgets C = {1, 5, 10, 25, 50} %,
// expected calibration error, forecast error) and Sec. 2.2 (Brier score and CRPS of the predicted
// distribution against the measured bin).  Where the paper is silent: Top_c is the first
// ceil(c n / 100) candidates (at least one) by decreasing expected speedup, lower index first on
// ties; the calibration buckets are ten equal-width confidence intervals (0, 0.1], ..., (0.9, 1]
// with a confidence of 0 in the first; the predicted bin is the arg max of p, lowest bin on ties.
#include <algorithm>
#include <cmath>
#include <numeric>
#include <vector>

#include "gf.h"
#include "kernels.h"

namespace {
constexpr double kUpperEdges[7] = {0.25, 0.5, 0.71, 1.0, 1.41, 2.0, 4.0};
constexpr int kBudgets[5] = {1, 5, 10, 25, 50};
}  // namespace

extern "C" int gf_speedup_bin(double S) {
  for (int b = 0; b < 7; ++b)
    if (S <= kUpperEdges[b]) return b + 1;
  return 8;
}

extern "C" int gf_score_forecasts(int32_t n, const double* p, const double* S, const double* m_bins,
                                  double* scores) {
  if (n < 1 || !p || !S || !m_bins || !scores) {
    gf::set_error_short("bad argument");
    return GF_EINVAL;
  }
  for (int64_t i = 0; i < (int64_t)n * 8; ++i)
    if (!(p[i] >= 0.0) || !std::isfinite(p[i])) {
      gf::set_error_short("bad p");
      return GF_EINVAL;
    }
  for (int32_t i = 0; i < n; ++i)
    if (!(S[i] > 0.0) || !std::isfinite(S[i])) {
      gf::set_error_short("bad speedup");
      return GF_EINVAL;
    }
  // expected speedups and the ranking they give
  std::vector<double> s_hat(n);
  for (int32_t i = 0; i < n; ++i) {
    double acc = 0.0;
    for (int b = 0; b < 8; ++b) acc += p[(int64_t)i * 8 + b] * m_bins[b];
    s_hat[i] = acc;
  }
  std::vector<int32_t> order(n);
  std::iota(order.begin(), order.end(), 0);
  std::stable_sort(order.begin(), order.end(), [&](int32_t a, int32_t b) { return s_hat[a] > s_hat[b]; });
  const double best = *std::max_element(S, S + n);
  double rec = 0.0;
  for (int c : kBudgets) {
    const int32_t k = std::max<int32_t>(1, (int32_t)std::ceil(c * (double)n / 100.0));
    double top = 0.0;
    for (int32_t j = 0; j < k; ++j) top = std::max(top, S[order[j]]);
    rec += top / best;
  }
  rec *= 100.0 / 5.0;
  // per item: predicted bin (arg max, lowest on ties), confidence, measured bin
  double ece_num[10] = {0}, ece_conf[10] = {0}, ece_cnt[10] = {0};
  double ferr = 0.0, brier = 0.0, crps = 0.0;
  for (int32_t i = 0; i < n; ++i) {
    const double* pi = p + (int64_t)i * 8;
    int pred = 0;
    for (int b = 1; b < 8; ++b)
      if (pi[b] > pi[pred]) pred = b;
    const double conf = pi[pred];
    const int y = gf_speedup_bin(S[i]) - 1;
    const int bucket = std::min(9, std::max(0, (int)std::ceil(conf * 10.0) - 1));
    ece_cnt[bucket] += 1.0;
    ece_conf[bucket] += conf;
    ece_num[bucket] += pred == y ? 1.0 : 0.0;
    ferr += std::fabs(m_bins[pred] - S[i]);
    double bs = 0.0, cdf = 0.0, cr = 0.0;
    for (int b = 0; b < 8; ++b) {
      const double d = pi[b] - (b == y ? 1.0 : 0.0);
      bs += d * d;
      if (b < 7) {
        cdf += pi[b];
        const double t = cdf - (y <= b ? 1.0 : 0.0);
        cr += t * t;
      }
    }
    brier += 0.5 * bs;
    crps += cr / 7.0;
  }
  double ece = 0.0;
  for (int k = 0; k < 10; ++k)
    if (ece_cnt[k] > 0) ece += ece_cnt[k] / n * std::fabs(ece_num[k] / ece_cnt[k] - ece_conf[k] / ece_cnt[k]);
  scores[0] = rec;
  scores[1] = ece;
  scores[2] = ferr / n;
  scores[3] = brier / n;
  scores[4] = crps / n;
  return GF_OK;
}
