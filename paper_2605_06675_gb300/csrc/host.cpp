// Host half of librq: distortion-model fit, integer and continuous bit
// allocation, packed layout. Pure C++17, no CUDA.
//
// RateQuant (arXiv 2605.06675):
//   Assumption 1        D(b) = alpha * beta^-b
//   Alg. 1 stage 2      least squares of ln D on b at b = 2..6
//   App. W              poor fits (R^2 < 0.96) fall back to min(beta, beta_bar)
//   Eq. 1               min sum w_i D_i(b_i), sum b_i = B, bounds
//   Alg. 2, Prop. 3     greedy max-heap on marginal gain, optimal for convex D
//   Thm. 1, App. B.1    continuous reverse waterfilling with iterative clipping
#include <algorithm>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <limits>
#include <queue>
#include <vector>

#include "rq.h"

namespace {

bool is_contiguous_mask(uint32_t mask, int* lo, int* hi) {
  int first = -1, last = -1;
  for (int k = 1; k <= 8; ++k)
    if ((mask >> k) & 1u) {
      if (first < 0) first = k;
      last = k;
    }
  if (first < 0) return false;
  *lo = first;
  *hi = last;
  for (int k = first; k <= last; ++k)
    if (!((mask >> k) & 1u)) return false;
  return true;
}

// w alpha beta^-b, evaluated as ((w * alpha) * beta^-b)
inline double component_cost(double w, double a, double beta, int b) {
  return (w * a) * std::pow(beta, -static_cast<double>(b));
}

// gain of the (b+1)-th bit: w alpha beta^-b (1 - 1/beta)
inline double marginal_gain(double w, double a, double beta, int b) {
  return ((w * a) * std::pow(beta, -static_cast<double>(b))) * (1.0 - 1.0 / beta);
}

struct HeapItem {
  double gain;
  int32_t index;
};
// std::priority_queue pops the "largest"; larger gain first, then lower index
struct HeapOrder {
  bool operator()(const HeapItem& a, const HeapItem& b) const {
    if (a.gain != b.gain) return a.gain < b.gain;
    return a.index > b.index;
  }
};

rq_status greedy_alloc(int32_t n, const std::vector<double>& w, const double* alpha,
                       const double* beta, int64_t B, int lo, int hi, uint8_t* bits) {
  if (B < static_cast<int64_t>(n) * lo || B > static_cast<int64_t>(n) * hi)
    return RQ_ERR_INFEASIBLE;
  for (int32_t i = 0; i < n; ++i) bits[i] = static_cast<uint8_t>(lo);
  int64_t remaining = B - static_cast<int64_t>(n) * lo;
  std::priority_queue<HeapItem, std::vector<HeapItem>, HeapOrder> heap;
  if (lo < hi)
    for (int32_t i = 0; i < n; ++i) heap.push({marginal_gain(w[i], alpha[i], beta[i], lo), i});
  while (remaining > 0) {
    HeapItem top = heap.top();
    heap.pop();
    const int32_t i = top.index;
    bits[i] = static_cast<uint8_t>(bits[i] + 1);
    --remaining;
    if (bits[i] < hi) heap.push({marginal_gain(w[i], alpha[i], beta[i], bits[i]), i});
  }
  return RQ_OK;
}

// Exact optimum for any allowed set: suffix table g[i][r] = least cost of
// components i..n-1 spending r bits above the smallest allowed width. Only two
// rows of g are kept; choice[i][r] records the width that attains g[i][r]
// (the largest one on a tie, as the reconstruction has always taken it), and
// the bits are read off the choices from (0, R).
rq_status dp_alloc(int32_t n, const std::vector<double>& w, const double* alpha,
                   const double* beta, int64_t B, uint32_t mask, uint8_t* bits) {
  std::vector<int> widths;
  for (int k = 1; k <= 8; ++k)
    if ((mask >> k) & 1u) widths.push_back(k);
  const int lo = widths.front();
  const int64_t R = B - static_cast<int64_t>(n) * lo;
  if (R < 0) return RQ_ERR_INFEASIBLE;
  if (static_cast<double>(n + 1) * static_cast<double>(R + 1) > 4.0e8) return RQ_ERR_INVALID_ARG;
  const double inf = std::numeric_limits<double>::infinity();
  const size_t W = static_cast<size_t>(R + 1);
  std::vector<double> cur(W, inf), next(W, inf);
  std::vector<uint8_t> choice(static_cast<size_t>(n) * W, 0);
  next[0] = 0.0;                                  // g[n][r]: nothing left to spend
  const size_t nw = widths.size();
  for (int32_t i = n - 1; i >= 0; --i) {
    // g[i][r] = min over widths k of cost_k + g[i+1][r - (w_k - lo)]: one
    // branch-free pass per width over the shifted row; visiting the widths in
    // ascending order with <= keeps the largest width on a tie
    uint8_t* ch = &choice[static_cast<size_t>(i) * W];
    std::fill(cur.begin(), cur.end(), inf);
    for (size_t k = 0; k < nw; ++k) {
      const int64_t dlt = widths[k] - lo;
      const double c = component_cost(w[i], alpha[i], beta[i], widths[k]);
      const uint8_t kk = static_cast<uint8_t>(k);
      for (int64_t r = dlt; r <= R; ++r) {
        const double v = c + next[r - dlt];
        const bool take = v <= cur[r] && v != inf;
        cur[r] = take ? v : cur[r];
        ch[r] = take ? kk : ch[r];
      }
    }
    cur.swap(next);
  }
  if (next[R] == inf) return RQ_ERR_INFEASIBLE;
  int64_t r = R;
  for (int32_t i = 0; i < n; ++i) {
    const int k = choice[static_cast<size_t>(i) * W + r];
    bits[i] = static_cast<uint8_t>(widths[k]);
    r -= widths[k] - lo;
  }
  return r == 0 ? RQ_OK : RQ_ERR_INFEASIBLE;
}

}  // namespace

// ------------------------------------------------------ Lloyd-Max codebook ----
// The 2^b-level Lloyd-Max quantizer of a unit Gaussian (App. F Table 8;
// TurboQuant's scalar quantizer): levels that are the centroids of their
// nearest-level cells. Only the upper half is solved (the codebook is
// symmetric): Lloyd's iteration, then Newton's method on the fixed point
// (tridiagonal Jacobian: the centroid of cell i moves with its two edges,
// dC/dt = phi(t) (C - t) / p at the lower edge and phi(t) (t - C) / p at the
// upper one, each edge the midpoint of two levels).
namespace {

double gauss_pdf(double t) { return std::exp(-0.5 * t * t) * 0.3989422804014327; }
// P(X > t) for t >= 0 without cancellation
double gauss_tail(double t) { return 0.5 * std::erfc(t * 0.7071067811865476); }

// positive levels y[0] < ... < y[m-1] of the 2m-level codebook; the cells are
// [0, t_1), [t_1, t_2), ..., [t_{m-1}, inf) with t_k = (y[k-1] + y[k]) / 2
void lm_centroids(const std::vector<double>& y, std::vector<double>& c, std::vector<double>& ga,
                  std::vector<double>& gc) {
  const size_t m = y.size();
  for (size_t k = 0; k < m; ++k) {
    const double a = k == 0 ? 0.0 : 0.5 * (y[k - 1] + y[k]);
    const bool last = k + 1 == m;
    const double hi = last ? 0.0 : 0.5 * (y[k] + y[k + 1]);
    const double p = gauss_tail(a) - (last ? 0.0 : gauss_tail(hi));
    const double cc = (gauss_pdf(a) - (last ? 0.0 : gauss_pdf(hi))) / p;
    c[k] = cc;
    ga[k] = k == 0 ? 0.0 : gauss_pdf(a) * (cc - a) / p;      // the cell at 0 has a fixed edge
    gc[k] = last ? 0.0 : gauss_pdf(hi) * (hi - cc) / p;
  }
}

std::vector<double> lloyd_max_positive(int b) {
  const size_t m = static_cast<size_t>(1) << (b - 1);
  std::vector<double> y(m), c(m), ga(m), gc(m);
  // start: equally spaced over [0, 4]
  for (size_t k = 0; k < m; ++k) y[k] = 4.0 * (k + 0.5) / m;
  for (int it = 0; it < 400; ++it) {
    lm_centroids(y, c, ga, gc);
    y = c;
  }
  std::vector<double> lo(m), di(m), up(m), r(m), cp(m), dp(m), x(m);
  for (int it = 0; it < 60; ++it) {
    lm_centroids(y, c, ga, gc);
    for (size_t k = 0; k < m; ++k) {
      r[k] = c[k] - y[k];                        // Newton: (I - dC) step = C - y
      di[k] = 1.0 - 0.5 * (ga[k] + gc[k]);
      lo[k] = k ? -0.5 * ga[k] : 0.0;
      up[k] = k + 1 < m ? -0.5 * gc[k] : 0.0;
    }
    // at the centre cell the lower edge is 0 for every level set (symmetry)
    if (m > 0) di[0] = 1.0 - 0.5 * gc[0];
    cp[0] = m > 1 ? up[0] / di[0] : 0.0;
    dp[0] = r[0] / di[0];
    for (size_t k = 1; k < m; ++k) {
      const double den = di[k] - lo[k] * cp[k - 1];
      cp[k] = k + 1 < m ? up[k] / den : 0.0;
      dp[k] = (r[k] - lo[k] * dp[k - 1]) / den;
    }
    x[m - 1] = dp[m - 1];
    for (size_t k = m - 1; k-- > 0;) x[k] = dp[k] - cp[k] * x[k + 1];
    double big = 0.0;
    for (size_t k = 0; k < m; ++k) {
      y[k] += x[k];
      big = std::max(big, std::fabs(x[k]));
    }
    if (big < 1e-15) break;
  }
  return y;
}

// round to nearest fp16, ties to even (|v| within the fp16 normal range)
uint16_t to_half_bits(double v) {
  const uint16_t sign = v < 0 ? 0x8000u : 0u;
  const double a = std::fabs(v);
  if (a == 0.0) return sign;
  int e = 0;
  std::frexp(a, &e);                              // a = f 2^e, f in [0.5, 1)
  int E = e - 1;                                  // a = g 2^E, g in [1, 2)
  if (E < -14) E = -14;                           // subnormal range: fixed step 2^-24
  double mant = std::nearbyint(std::ldexp(a, 10 - E));     // rounds half to even
  if (mant >= 2048.0) {
    mant /= 2.0;
    ++E;
  }
  if (mant < 1024.0) return static_cast<uint16_t>(sign | static_cast<uint16_t>(mant));
  return static_cast<uint16_t>(sign | ((E + 15) << 10) | (static_cast<uint16_t>(mant) - 1024u));
}

struct LMCodebooks {
  uint16_t lv[8][256];
  LMCodebooks() {
    for (int b = 1; b <= 8; ++b) {
      const std::vector<double> y = lloyd_max_positive(b);
      const int m = 1 << (b - 1);
      for (int k = 0; k < m; ++k) {
        lv[b - 1][m + k] = to_half_bits(y[k]);
        lv[b - 1][m - 1 - k] = to_half_bits(-y[k]);
      }
    }
  }
};

}  // namespace

namespace rq {
// fp16 bit patterns of the 2^b levels, ascending (computed once, on first use)
const uint16_t* lloydmax_levels(int b) {
  static const LMCodebooks books;
  return books.lv[b - 1];
}
}  // namespace rq

extern "C" {

const char* rq_status_string(rq_status s) {
  switch (s) {
    case RQ_OK: return "ok";
    case RQ_ERR_INVALID_ARG: return "invalid argument";
    case RQ_ERR_INFEASIBLE: return "budget not reachable with the allowed bit-widths";
    case RQ_ERR_SHAPE: return "unsupported shape";
    case RQ_ERR_ALIGNMENT: return "device pointer not 16-byte aligned";
    case RQ_ERR_WORKSPACE: return "workspace too small";
    case RQ_ERR_CUDA: return "CUDA error";
  }
  return "unknown status";
}

int32_t rq_abi_version(void) { return RQ_ABI_VERSION; }

rq_status rq_lloydmax_levels(int32_t b, uint16_t* levels) {
  if (b < 1 || b > 8 || !levels) return RQ_ERR_INVALID_ARG;
  std::memcpy(levels, rq::lloydmax_levels(b), sizeof(uint16_t) << b);
  return RQ_OK;
}

rq_status rq_fit_distortion(int32_t n, const double* mse, int32_t b_lo, int32_t b_hi,
                            double r2_min, const int32_t* classes, double* alpha, double* beta,
                            double* r2) {
  if (n <= 0 || !mse || !alpha || !beta || !r2) return RQ_ERR_INVALID_ARG;
  if (b_lo < 1 || b_hi > 8 || b_lo >= b_hi) return RQ_ERR_INVALID_ARG;
  const double inf = std::numeric_limits<double>::infinity();
  for (int32_t i = 0; i < n; ++i) {
    double xs[8], ys[8];
    int m = 0;
    for (int b = b_lo; b <= b_hi; ++b) {
      const double D = mse[static_cast<size_t>(i) * 8 + (b - 1)];
      if (D > 0.0) {
        xs[m] = static_cast<double>(b);
        ys[m] = std::log(D);
        ++m;
      }
    }
    if (m < 2) {
      alpha[i] = 0.0;
      beta[i] = inf;
      r2[i] = 1.0;
      continue;
    }
    double sx = 0.0, sy = 0.0;
    for (int k = 0; k < m; ++k) {
      sx += xs[k];
      sy += ys[k];
    }
    const double mx = sx / m, my = sy / m;
    double sxy = 0.0, sxx = 0.0;
    for (int k = 0; k < m; ++k) {
      sxy += (xs[k] - mx) * (ys[k] - my);
      sxx += (xs[k] - mx) * (xs[k] - mx);
    }
    const double slope = sxy / sxx;
    const double icept = my - slope * mx;
    double ss_res = 0.0, ss_tot = 0.0;
    for (int k = 0; k < m; ++k) {
      const double res = ys[k] - (icept + slope * xs[k]);
      ss_res += res * res;
      ss_tot += (ys[k] - my) * (ys[k] - my);
    }
    alpha[i] = std::exp(icept);
    beta[i] = std::exp(-slope);
    r2[i] = (ss_tot == 0.0) ? (ss_res == 0.0 ? 1.0 : 0.0) : 1.0 - ss_res / ss_tot;
  }
  if (r2_min > 0.0) {
    // class means of the fitted (finite) beta, before any fallback
    std::vector<int32_t> cls(n, 0);
    if (classes)
      for (int32_t i = 0; i < n; ++i) cls[i] = classes[i];
    std::vector<int32_t> keys;
    for (int32_t i = 0; i < n; ++i) {
      bool seen = false;
      for (int32_t k : keys) seen = seen || (k == cls[i]);
      if (!seen) keys.push_back(cls[i]);
    }
    std::vector<double> fitted(beta, beta + n);
    for (int32_t key : keys) {
      double s = 0.0;
      int cnt = 0;
      for (int32_t i = 0; i < n; ++i)
        if (cls[i] == key && std::isfinite(fitted[i])) {
          s += fitted[i];
          ++cnt;
        }
      const double mean = cnt > 0 ? s / cnt : inf;
      for (int32_t i = 0; i < n; ++i)
        if (cls[i] == key && r2[i] < r2_min) beta[i] = std::fmin(fitted[i], mean);
    }
  }
  return RQ_OK;
}

rq_status rq_alloc(int32_t n, const double* w, const double* alpha, const double* beta,
                   double avg_bits, uint32_t allowed_mask, uint32_t flags, uint8_t* bits_out,
                   double* objective_out) {
  if (n <= 0 || !w || !alpha || !beta || !bits_out) return RQ_ERR_INVALID_ARG;
  if ((allowed_mask & 0x1FEu) == 0 || (allowed_mask & ~0x1FEu) != 0) return RQ_ERR_INVALID_ARG;
  if (!std::isfinite(avg_bits)) return RQ_ERR_INVALID_ARG;
  std::vector<double> wv(w, w + n);
  if (flags & RQ_CAP_5X) {
    double mean = 0.0;
    for (int32_t i = 0; i < n; ++i) mean += wv[i];
    mean /= n;
    for (int32_t i = 0; i < n; ++i) wv[i] = std::fmin(wv[i], 5.0 * mean);
  }
  const int64_t B = static_cast<int64_t>(std::floor(avg_bits * n + 0.5));
  int lo = 0, hi = 0;
  rq_status st = is_contiguous_mask(allowed_mask, &lo, &hi)
                     ? greedy_alloc(n, wv, alpha, beta, B, lo, hi, bits_out)
                     : dp_alloc(n, wv, alpha, beta, B, allowed_mask, bits_out);
  if (st != RQ_OK) return st;
  if (objective_out) {
    double J = 0.0;
    for (int32_t i = 0; i < n; ++i) J += component_cost(wv[i], alpha[i], beta[i], bits_out[i]);
    *objective_out = J;
  }
  return RQ_OK;
}

rq_status rq_alloc_continuous(int32_t n, const double* w, const double* alpha,
                              const double* beta, double avg_bits, double b_min, double b_max,
                              double* b_out) {
  if (n <= 0 || !w || !alpha || !beta || !b_out) return RQ_ERR_INVALID_ARG;
  if (!(b_min <= b_max)) return RQ_ERR_INVALID_ARG;
  for (int32_t i = 0; i < n; ++i)
    if (!(w[i] > 0.0) || !(alpha[i] > 0.0) || !(beta[i] > 1.0)) return RQ_ERR_INVALID_ARG;
  const double B = avg_bits * n;
  if (B < n * b_min - 1e-9 || B > n * b_max + 1e-9) return RQ_ERR_INFEASIBLE;
  // ln of w alpha ln(beta), and ln(beta)
  std::vector<double> A(n), lb(n);
  for (int32_t i = 0; i < n; ++i) {
    A[i] = std::log(w[i] * alpha[i] * std::log(beta[i]));
    lb[i] = std::log(beta[i]);
  }
  std::vector<char> fixed(n, 0);
  std::vector<double> fixed_val(n, 0.0);
  for (int32_t round = 0; round <= n; ++round) {
    double Bf = B;
    bool any_free = false;
    for (int32_t i = 0; i < n; ++i) {
      if (fixed[i]) Bf -= fixed_val[i];
      else any_free = true;
    }
    if (!any_free) break;
    // sum_F (A_i - ln lambda) / ln beta_i = B_F  ->  ln lambda in closed form
    double num = 0.0, den = 0.0;
    for (int32_t i = 0; i < n; ++i)
      if (!fixed[i]) {
        num += A[i] / lb[i];
        den += 1.0 / lb[i];
      }
    const double ln_lambda = (num - Bf) / den;
    bool changed = false;
    for (int32_t i = 0; i < n; ++i) {
      if (fixed[i]) continue;
      const double b = (A[i] - ln_lambda) / lb[i];
      if (b < b_min) {
        fixed[i] = 1;
        fixed_val[i] = b_min;
        changed = true;
      } else if (b > b_max) {
        fixed[i] = 1;
        fixed_val[i] = b_max;
        changed = true;
      } else {
        b_out[i] = b;
      }
    }
    if (!changed) break;
  }
  for (int32_t i = 0; i < n; ++i)
    if (fixed[i]) b_out[i] = fixed_val[i];
  return RQ_OK;
}

rq_status rq_packed_layout(const rq_cache_desc* desc, const uint8_t* bits, uint64_t* offsets,
                           uint64_t* total_bytes) {
  if (!desc || !bits || !total_bytes) return RQ_ERR_INVALID_ARG;
  if (desc->L <= 0 || desc->B < 0 || desc->H_kv <= 0 || desc->S < 0) return RQ_ERR_INVALID_ARG;
  if (desc->d != RQ_HEAD_DIM || desc->group != RQ_GROUP || desc->S % RQ_GROUP != 0)
    return RQ_ERR_SHAPE;
  const uint64_t nblk = static_cast<uint64_t>(desc->S / RQ_GROUP);
  uint64_t pos = 0;
  for (int32_t l = 0; l < desc->L; ++l)
    for (int32_t b = 0; b < desc->B; ++b)
      for (int32_t h = 0; h < desc->H_kv; ++h)
        for (int32_t kind = 0; kind < 2; ++kind) {
          const int bw = bits[(static_cast<size_t>(l) * desc->H_kv + h) * 2 + kind];
          if (bw < 1 || bw > 8) return RQ_ERR_INVALID_ARG;
          if (offsets)
            offsets[((static_cast<size_t>(l) * desc->B + b) * desc->H_kv + h) * 2 + kind] = pos;
          pos += nblk * 512ull * static_cast<uint64_t>(bw + 1);
        }
  *total_bytes = pos;
  return RQ_OK;
}

}  // extern "C"
