// Host side of libcobra: allocation (C1, C2 damped update, exact DP), calibration helpers
// (covariance, symmetric eigen-decomposition, attention-KL weights, Hadamard fusion,
// loading factor), cache layout and the device parameter block.
//
// Floating-point sums in the allocator run sequentially in head / index order, and this
// file is compiled without FMA contraction, so the allocator's results are reproducible
// bit for bit by any implementation that follows the same order.
#include <algorithm>
#include <cstddef>
#include <cmath>
#include <cstring>
#include <limits>
#include <numeric>
#include <vector>

#include <cuda_runtime.h>

#include "../../include/cobra.h"
#include "internal.h"

using cobra::align_up;

extern "C" int cobra_version(void) { return COBRA_VERSION; }

extern "C" const char* cobra_status_string(int s) {
  switch (s) {
    case COBRA_OK: return "ok";
    case COBRA_EINVAL: return "invalid argument";
    case COBRA_EALIGN: return "misaligned pointer or offset";
    case COBRA_EBUDGET: return "infeasible budget";
    case COBRA_ECUDA: return "CUDA error";
    case COBRA_ETIMEOUT: return "device wait timed out";
    case COBRA_ESPACE: return "buffer too small";
    default: return "unknown status";
  }
}

// ----------------------------------------------------------------------------------------
// Allocation.  Eq. (drb-preview) D(r, b) = sum_{i>r} w_i + q(b) sum_{i<=r} w_i, Eq. (q)
// q(b) = 2^{-2b} / 12; C1 (Sec. 3.2) enumerates the feasible (r, b) with r*b <= B; C2 (App. D,
// Eq. c2-update) moves budgets by eta * Bbar * (sqrt(D_h / Dbar) - 1) and renormalises.
// ----------------------------------------------------------------------------------------
namespace {

struct Opts {
  int mode, rounds, b_min, b_max, r_step, allow_r0, complete;
  double eta, B_min;
};

double qdist(int b) { return std::ldexp(1.0, -2 * b) / 12.0; }

struct Head {
  std::vector<double> pre;  // pre[k] = w_0 + ... + w_{k-1}
  int d;
};

double distortion(const Head& h, int r, int b) {
  if (r == 0) return h.pre[h.d];
  return (h.pre[h.d] - h.pre[r]) + qdist(b) * h.pre[r];
}

std::vector<int> rank_grid(int d, const Opts& o) {
  std::vector<int> g;
  if (o.allow_r0) g.push_back(0);
  for (int r = o.r_step; r <= d; r += o.r_step) g.push_back(r);
  return g;
}

struct Choice {
  int r = 0, b = 0;
  double D = 0.0;
  bool ok = false;
};

// C1: smallest D; ties -> smaller r*b, then larger r.
Choice c1(const Head& h, double B, const Opts& o, const std::vector<int>& grid) {
  Choice best;
  long long best_rb = 0;
  for (int r : grid) {
    int b;
    if (r == 0) {
      b = 0;
    } else {
      double f = std::floor(B / (double)r);
      b = f >= (double)o.b_max ? o.b_max : (int)f;
      if (b < o.b_min) continue;
    }
    double D = distortion(h, r, b);
    long long rb = (long long)r * b;
    bool better = !best.ok || D < best.D || (D == best.D && (rb < best_rb || (rb == best_rb && r > best.r)));
    if (better) {
      best.r = r;
      best.b = b;
      best.D = D;
      best.ok = true;
      best_rb = rb;
    }
  }
  return best;
}

struct Upgrade {
  double gain = -1.0;
  long long extra = 0;
  int r = 0, b = 0;
  double D = 0.0;
  bool valid = false;  // computed
};

Upgrade best_upgrade(const Head& h, int r0, int b0, double D0, long long slack, const Opts& o,
                     const std::vector<int>& grid) {
  Upgrade best;
  best.valid = true;
  bool have = false;
  for (int r : grid) {
    if (r == 0) continue;
    for (int b = o.b_min; b <= o.b_max; ++b) {
      long long extra = (long long)r * b - (long long)r0 * b0;
      if (extra <= 0 || extra > slack) continue;
      double D = distortion(h, r, b);
      if (!(D < D0)) continue;
      double gain = (D0 - D) / (double)extra;
      if (!have || gain > best.gain) {
        best.gain = gain;
        best.extra = extra;
        best.r = r;
        best.b = b;
        best.D = D;
        have = true;
      }
    }
  }
  if (!have) {
    best.gain = -1.0;
    best.extra = 0;
  }
  return best;
}

long long complete_alloc(const std::vector<Head>& H, std::vector<int>& r, std::vector<int>& b,
                         std::vector<double>& D, double B_tot, const Opts& o, const std::vector<int>& grid) {
  const int n = (int)H.size();
  long long used = 0;
  for (int h = 0; h < n; ++h) used += (long long)r[h] * b[h];
  long long slack = (long long)std::floor(B_tot + 1e-9) - used;
  std::vector<Upgrade> cache(n);
  while (slack > 0) {
    int best_h = -1;
    double best_gain = 0.0;
    for (int h = 0; h < n; ++h) {
      if (!cache[h].valid || cache[h].extra > slack)
        cache[h] = best_upgrade(H[h], r[h], b[h], D[h], slack, o, grid);
      const Upgrade& c = cache[h];
      if (c.gain <= 0) continue;
      if (best_h < 0 || c.gain > best_gain) {
        best_gain = c.gain;
        best_h = h;
      }
    }
    if (best_h < 0) break;
    const Upgrade c = cache[best_h];
    r[best_h] = c.r;
    b[best_h] = c.b;
    D[best_h] = c.D;
    slack -= c.extra;
    cache[best_h].valid = false;
  }
  return slack;
}

// Exact DP over integer rates (App. E separable knapsack), on per-head options.
struct RateOpt {
  long long rate;
  double D;
  int r, b;
};

// One option per distinct rate: the smallest D, the first in the given order on ties; sorted
// by rate.
std::vector<RateOpt> unique_by_rate(const std::vector<RateOpt>& all) {
  std::vector<RateOpt> uniq;
  for (const RateOpt& x : all) {
    bool found = false;
    for (RateOpt& u : uniq)
      if (u.rate == x.rate) {
        found = true;
        if (x.D < u.D) u = x;
        break;
      }
    if (!found) uniq.push_back(x);
  }
  std::stable_sort(uniq.begin(), uniq.end(), [](const RateOpt& a, const RateOpt& c) { return a.rate < c.rate; });
  return uniq;
}

cobra_status dp_over_options(const std::vector<std::vector<RateOpt>>& opts, double B_tot, std::vector<int>& r,
                             std::vector<int>& b, std::vector<double>& D) {
  const int n = (int)opts.size();
  const long long cap = (long long)std::floor(B_tot + 1e-9);
  if (cap < 0 || cap > (1LL << 26)) return COBRA_EINVAL;
  for (const auto& o : opts)
    if (o.size() > 32767) return COBRA_EINVAL;
  const double INF = std::numeric_limits<double>::infinity();
  std::vector<double> dp(cap + 1, INF), nw(cap + 1);
  dp[0] = 0.0;
  std::vector<int16_t> choice((size_t)n * (cap + 1), -1);
  for (int h = 0; h < n; ++h) {
    std::fill(nw.begin(), nw.end(), INF);
    int16_t* ch = choice.data() + (size_t)h * (cap + 1);
    for (size_t k = 0; k < opts[h].size(); ++k) {
      const RateOpt& x = opts[h][k];
      if (x.rate > cap) break;
      for (long long beta = x.rate; beta <= cap; ++beta) {
        double cand = dp[beta - x.rate] + x.D;
        if (cand < nw[beta]) {
          nw[beta] = cand;
          ch[beta] = (int16_t)k;
        }
      }
    }
    dp.swap(nw);
  }
  long long beta = 0;
  for (long long k = 1; k <= cap; ++k)
    if (dp[k] < dp[beta]) beta = k;
  if (!(dp[beta] < INF)) return COBRA_EBUDGET;
  for (int h = n - 1; h >= 0; --h) {
    int k = choice[(size_t)h * (cap + 1) + beta];
    if (k < 0) return COBRA_EBUDGET;
    const RateOpt& x = opts[h][k];
    r[h] = x.r;
    b[h] = x.b;
    D[h] = x.D;
    beta -= x.rate;
  }
  return COBRA_OK;
}

// the surrogate's options: every (r, b) of the grid, D from Eq. drb-preview
cobra_status exact_dp(const std::vector<Head>& H, double B_tot, const Opts& o, const std::vector<int>& grid,
                      std::vector<int>& r, std::vector<int>& b, std::vector<double>& D) {
  const int n = (int)H.size();
  std::vector<std::vector<RateOpt>> opts(n);
  for (int h = 0; h < n; ++h) {
    std::vector<RateOpt> all;
    for (int rr : grid) {
      if (rr == 0) {
        all.push_back({0, distortion(H[h], 0, 0), 0, 0});
        continue;
      }
      for (int bb = o.b_min; bb <= o.b_max; ++bb) all.push_back({(long long)rr * bb, distortion(H[h], rr, bb), rr, bb});
    }
    opts[h] = unique_by_rate(all);
  }
  return dp_over_options(opts, B_tot, r, b, D);
}

}  // namespace

extern "C" cobra_status cobra_allocate_tables(int n_heads, int d, int n_r, const int* r_list, int n_b,
                                              const int* b_list, const double* D, double bpd, int* r_out, int* b_out,
                                              double* dist, long long* rate_bits) {
  if (n_heads <= 0 || d <= 0 || d > 4096 || n_r <= 0 || n_b <= 0 || !r_list || !b_list || !D || !r_out || !b_out ||
      !(bpd >= 0.0) || !std::isfinite(bpd))
    return COBRA_EINVAL;
  for (int i = 0; i < n_r; ++i)
    if (r_list[i] < 0 || r_list[i] > d || (i > 0 && r_list[i] <= r_list[i - 1])) return COBRA_EINVAL;
  for (int j = 0; j < n_b; ++j)
    if (b_list[j] < 1 || b_list[j] > 16 || (j > 0 && b_list[j] <= b_list[j - 1])) return COBRA_EINVAL;
  for (long long k = 0; k < (long long)n_heads * n_r * n_b; ++k)
    if (!std::isfinite(D[k])) return COBRA_EINVAL;
  std::vector<std::vector<RateOpt>> opts(n_heads);
  for (int h = 0; h < n_heads; ++h) {
    std::vector<RateOpt> all;
    for (int i = 0; i < n_r; ++i) {
      const double* row = D + ((size_t)h * n_r + i) * n_b;
      if (r_list[i] == 0) {
        all.push_back({0, row[0], 0, 0});
        continue;
      }
      for (int j = 0; j < n_b; ++j) all.push_back({(long long)r_list[i] * b_list[j], row[j], r_list[i], b_list[j]});
    }
    opts[h] = unique_by_rate(all);
  }
  std::vector<int> r(n_heads), b(n_heads);
  std::vector<double> Dh(n_heads);
  const double B_tot = (double)((long long)n_heads * d) * bpd;
  cobra_status st = dp_over_options(opts, B_tot, r, b, Dh);
  if (st != COBRA_OK) return st;
  long long used = 0;
  for (int h = 0; h < n_heads; ++h) {
    r_out[h] = r[h];
    b_out[h] = b[h];
    if (dist) dist[h] = Dh[h];
    used += (long long)r[h] * b[h];
  }
  if (rate_bits) *rate_bits = used;
  return COBRA_OK;
}

extern "C" void cobra_alloc_opts_default(cobra_alloc_opts* o) {
  if (!o) return;
  o->mode = COBRA_ALLOC_DAMPED;
  o->rounds = 5;
  o->eta = 0.3;
  o->b_min = 1;
  o->b_max = 8;
  o->r_step = 2;
  o->allow_r0 = 1;
  o->B_min = -1.0;
  o->complete = 1;
}

extern "C" cobra_status cobra_allocate(int n_heads, int d, const double* w, double bpd, const cobra_alloc_opts* opts,
                                       int* r_out, int* b_out, double* budget, double* dist, long long* rate_bits) {
  if (n_heads <= 0 || d <= 0 || d > 4096 || !w || !r_out || !b_out || !(bpd >= 0.0) || !std::isfinite(bpd))
    return COBRA_EINVAL;
  cobra_alloc_opts def;
  cobra_alloc_opts_default(&def);
  const cobra_alloc_opts& oo = opts ? *opts : def;
  if (oo.mode < 0 || oo.mode > 2 || oo.rounds < 0 || oo.b_min < 1 || oo.b_max > 16 || oo.b_min > oo.b_max ||
      oo.r_step < 1 || !std::isfinite(oo.eta))
    return COBRA_EINVAL;
  Opts o{oo.mode, oo.rounds, oo.b_min, oo.b_max, oo.r_step, oo.allow_r0 ? 1 : 0, oo.complete ? 1 : 0, oo.eta, oo.B_min};
  const double Bmin = o.B_min >= 0 ? o.B_min : (o.allow_r0 ? 0.0 : (double)(o.r_step * o.b_min));
  for (long long k = 0; k < (long long)n_heads * d; ++k)
    if (!std::isfinite(w[k])) return COBRA_EINVAL;

  std::vector<Head> H(n_heads);
  for (int h = 0; h < n_heads; ++h) {
    H[h].d = d;
    H[h].pre.assign(d + 1, 0.0);
    double s = 0.0;
    for (int i = 0; i < d; ++i) {
      s = s + w[(size_t)h * d + i];
      H[h].pre[i + 1] = s;
    }
  }
  const std::vector<int> grid = rank_grid(d, o);
  const double B_tot = (double)((long long)n_heads * d) * bpd;
  std::vector<int> r(n_heads), b(n_heads);
  std::vector<double> D(n_heads), B(n_heads, bpd * (double)d);

  if (o.mode == COBRA_ALLOC_EXACT) {
    cobra_status st = exact_dp(H, B_tot, o, grid, r, b, D);
    if (st != COBRA_OK) return st;
    for (int h = 0; h < n_heads; ++h) B[h] = (double)((long long)r[h] * b[h]);
  } else {
    if (o.mode == COBRA_ALLOC_DAMPED) {
      const double Bbar = B_tot / (double)n_heads;
      std::vector<double> Ds(n_heads), newB(n_heads);
      for (int round = 0; round < o.rounds; ++round) {
        for (int h = 0; h < n_heads; ++h) {
          Choice c = c1(H[h], B[h], o, grid);
          if (!c.ok) return COBRA_EBUDGET;
          Ds[h] = c.D;
        }
        double s = 0.0;
        for (int h = 0; h < n_heads; ++h) s = s + Ds[h];
        const double Dbar = s / (double)n_heads;
        if (Dbar == 0.0) break;
        for (int h = 0; h < n_heads; ++h) {
          double x = B[h] + o.eta * Bbar * (std::sqrt(Ds[h] / Dbar) - 1.0);
          newB[h] = x > Bmin ? x : Bmin;
        }
        s = 0.0;
        for (int h = 0; h < n_heads; ++h) s = s + newB[h];
        const double f = B_tot / s;
        for (int h = 0; h < n_heads; ++h) {
          double x = newB[h] * f;
          B[h] = x > Bmin ? x : Bmin;
        }
      }
    }
    for (int h = 0; h < n_heads; ++h) {
      Choice c = c1(H[h], B[h], o, grid);
      if (!c.ok) return COBRA_EBUDGET;
      r[h] = c.r;
      b[h] = c.b;
      D[h] = c.D;
    }
    if (o.complete) complete_alloc(H, r, b, D, B_tot, o, grid);
  }
  long long used = 0;
  for (int h = 0; h < n_heads; ++h) {
    r_out[h] = r[h];
    b_out[h] = b[h];
    if (budget) budget[h] = B[h];
    if (dist) dist[h] = D[h];
    used += (long long)r[h] * b[h];
  }
  if (rate_bits) *rate_bits = used;
  return COBRA_OK;
}

// ----------------------------------------------------------------------------------------
// Quantizer loading factor: minimise the exact MSE of the 2^b-cell clamped uniform quantizer
// on N(0, 1) over L (golden-section search).  Cell MSE closed form:
//   int_a^b (x - c)^2 phi = (1 + c^2)(Phi(b) - Phi(a)) - (b phi(b) - a phi(a)) + 2c (phi(b) - phi(a)).
// ----------------------------------------------------------------------------------------
namespace {
double nphi(double x) { return std::isinf(x) ? 0.0 : std::exp(-0.5 * x * x) / std::sqrt(2.0 * M_PI); }
double nPhi(double x) {
  if (x == INFINITY) return 1.0;
  if (x == -INFINITY) return 0.0;
  return 0.5 * std::erfc(-x / std::sqrt(2.0));
}
double cell_mse(double a, double b, double c) {
  double ta = std::isinf(a) ? 0.0 : a * nphi(a);
  double tb = std::isinf(b) ? 0.0 : b * nphi(b);
  return (1.0 + c * c) * (nPhi(b) - nPhi(a)) - (tb - ta) + 2.0 * c * (nphi(b) - nphi(a));
}
double gauss_mse(double L, int bits) {
  const int n = 1 << bits;
  const double step = 2.0 * L / n;
  double total = 0.0;
  for (int k = 0; k < n; ++k) {
    double lo = k == 0 ? -INFINITY : -L + k * step;
    double hi = k == n - 1 ? INFINITY : -L + (k + 1) * step;
    total += cell_mse(lo, hi, -L + (k + 0.5) * step);
  }
  return total;
}
}  // namespace

extern "C" cobra_status cobra_loading_factor(int b, double* L) {
  if (b < 1 || b > 8 || !L) return COBRA_EINVAL;
  const double gr = (std::sqrt(5.0) - 1.0) / 2.0;
  double a = 0.5, c = 8.0;
  double x1 = c - gr * (c - a), x2 = a + gr * (c - a);
  double f1 = gauss_mse(x1, b), f2 = gauss_mse(x2, b);
  while (c - a > 1e-12) {
    if (f1 <= f2) {
      c = x2;
      x2 = x1;
      f2 = f1;
      x1 = c - gr * (c - a);
      f1 = gauss_mse(x1, b);
    } else {
      a = x1;
      x1 = x2;
      f1 = f2;
      x2 = a + gr * (c - a);
      f2 = gauss_mse(x2, b);
    }
  }
  *L = 0.5 * (a + c);
  return COBRA_OK;
}

// ----------------------------------------------------------------------------------------
// Hadamard rotation (Sec. 3.4): blockdiag of normalised Sylvester blocks for the binary
// digits of r (largest first), columns multiplied by the sign flip.
// ----------------------------------------------------------------------------------------
extern "C" cobra_status cobra_hadamard(int r, const int8_t* signs, double* H) {
  if (r < 1 || r > 4096 || !signs || !H) return COBRA_EINVAL;
  for (int i = 0; i < r; ++i)
    if (signs[i] != 1 && signs[i] != -1) return COBRA_EINVAL;
  std::fill(H, H + (size_t)r * r, 0.0);
  int o = 0;
  for (int bit = 1 << 12; bit; bit >>= 1) {
    if (!(r & bit)) continue;
    const double s = 1.0 / std::sqrt((double)bit);
    for (int i = 0; i < bit; ++i)
      for (int j = 0; j < bit; ++j) {
        // Sylvester entry: (-1)^{popcount(i & j)}
        int par = __builtin_popcount((unsigned)(i & j)) & 1;
        H[(size_t)(o + i) * r + (o + j)] = (par ? -s : s) * (double)signs[o + j];
      }
    o += bit;
  }
  return COBRA_OK;
}

// ----------------------------------------------------------------------------------------
// Calibration: centred covariance, cyclic Jacobi eigen-decomposition, sign rule, KL weights.
// ----------------------------------------------------------------------------------------
namespace {
// Symmetric eigen-decomposition by cyclic Jacobi rotations.  A (n x n, row-major) is
// destroyed; on return lam holds the eigenvalues and V (row-major, column j = eigenvector j).
void jacobi_eigen(std::vector<double>& A, int n, std::vector<double>& lam, std::vector<double>& V) {
  V.assign((size_t)n * n, 0.0);
  for (int i = 0; i < n; ++i) V[(size_t)i * n + i] = 1.0;
  double scale = 0.0;
  for (size_t k = 0; k < A.size(); ++k) scale += A[k] * A[k];
  scale = std::sqrt(scale);
  for (int sweep = 0; sweep < 100; ++sweep) {
    double off = 0.0;
    for (int p = 0; p < n; ++p)
      for (int q = p + 1; q < n; ++q) off += A[(size_t)p * n + q] * A[(size_t)p * n + q];
    if (std::sqrt(off) <= 1e-15 * scale || off == 0.0) break;
    for (int p = 0; p < n; ++p) {
      for (int q = p + 1; q < n; ++q) {
        const double apq = A[(size_t)p * n + q];
        if (apq == 0.0) continue;
        const double app = A[(size_t)p * n + p], aqq = A[(size_t)q * n + q];
        const double theta = (aqq - app) / (2.0 * apq);
        const double t = (theta >= 0 ? 1.0 : -1.0) / (std::fabs(theta) + std::sqrt(theta * theta + 1.0));
        const double c = 1.0 / std::sqrt(t * t + 1.0), s = t * c;
        for (int k = 0; k < n; ++k) {  // columns p, q
          const double akp = A[(size_t)k * n + p], akq = A[(size_t)k * n + q];
          A[(size_t)k * n + p] = c * akp - s * akq;
          A[(size_t)k * n + q] = s * akp + c * akq;
        }
        for (int k = 0; k < n; ++k) {  // rows p, q
          const double apk = A[(size_t)p * n + k], aqk = A[(size_t)q * n + k];
          A[(size_t)p * n + k] = c * apk - s * aqk;
          A[(size_t)q * n + k] = s * apk + c * aqk;
        }
        A[(size_t)p * n + q] = 0.0;
        A[(size_t)q * n + p] = 0.0;
        for (int k = 0; k < n; ++k) {
          const double vkp = V[(size_t)k * n + p], vkq = V[(size_t)k * n + q];
          V[(size_t)k * n + p] = c * vkp - s * vkq;
          V[(size_t)k * n + q] = s * vkp + c * vkq;
        }
      }
    }
  }
  lam.resize(n);
  for (int i = 0; i < n; ++i) lam[i] = A[(size_t)i * n + i];
}
}  // namespace

extern "C" cobra_status cobra_calibrate_head(int n, int d, const float* x, int nq, const float* q, double* mu,
                                             double* lam_out, double* U_out, double* w_out) {
  if (n < 1 || d < 1 || d > 1024 || !x || !mu || !lam_out || !U_out || !w_out || nq < 0 || (nq > 0 && !q))
    return COBRA_EINVAL;
  std::vector<double> m(d, 0.0);
  for (int t = 0; t < n; ++t)
    for (int i = 0; i < d; ++i) m[i] += (double)x[(size_t)t * d + i];
  for (int i = 0; i < d; ++i) m[i] /= (double)n;
  std::vector<double> C((size_t)d * d, 0.0), xc(d);
  for (int t = 0; t < n; ++t) {
    for (int i = 0; i < d; ++i) xc[i] = (double)x[(size_t)t * d + i] - m[i];
    for (int i = 0; i < d; ++i) {
      const double a = xc[i];
      double* row = C.data() + (size_t)i * d;
      for (int j = i; j < d; ++j) row[j] += a * xc[j];
    }
  }
  for (int i = 0; i < d; ++i)
    for (int j = i; j < d; ++j) {
      C[(size_t)i * d + j] /= (double)n;
      C[(size_t)j * d + i] = C[(size_t)i * d + j];
    }
  std::vector<double> lam, V;
  jacobi_eigen(C, d, lam, V);
  std::vector<int> order(d);
  std::iota(order.begin(), order.end(), 0);
  std::stable_sort(order.begin(), order.end(), [&](int a, int b) { return lam[a] > lam[b]; });
  std::vector<double> L(d), U((size_t)d * d);  // U column-major
  for (int j = 0; j < d; ++j) {
    const int src = order[j];
    L[j] = lam[src];
    int kmax = 0;
    double vmax = -1.0;
    for (int i = 0; i < d; ++i) {
      double a = std::fabs(V[(size_t)i * d + src]);
      if (a > vmax) {
        vmax = a;
        kmax = i;
      }
    }
    const double sgn = V[(size_t)kmax * d + src] < 0 ? -1.0 : 1.0;
    for (int i = 0; i < d; ++i) U[(size_t)j * d + i] = sgn * V[(size_t)i * d + src];
  }
  std::vector<double> w(d);
  std::vector<int> perm(d);
  std::iota(perm.begin(), perm.end(), 0);
  if (nq > 0) {
    std::vector<double> sq(d, 0.0);
    for (int t = 0; t < nq; ++t) {
      const float* qt = q + (size_t)t * d;
      for (int j = 0; j < d; ++j) {
        const double* u = U.data() + (size_t)j * d;
        double p = 0.0;
        for (int i = 0; i < d; ++i) p += u[i] * (double)qt[i];
        sq[j] += p * p;
      }
    }
    for (int j = 0; j < d; ++j) w[j] = (sq[j] / (double)nq) * L[j];
    std::stable_sort(perm.begin(), perm.end(), [&](int a, int b) { return w[a] > w[b]; });
  } else {
    for (int j = 0; j < d; ++j) w[j] = L[j];
  }
  for (int i = 0; i < d; ++i) mu[i] = m[i];
  for (int j = 0; j < d; ++j) {
    const int src = perm[j];
    lam_out[j] = L[src];
    w_out[j] = w[src];
    std::memcpy(U_out + (size_t)j * d, U.data() + (size_t)src * d, sizeof(double) * d);
  }
  return COBRA_OK;
}

extern "C" cobra_status cobra_fuse_basis(int d, int r, int b, const double* U, const double* lam, const int8_t* signs,
                                         float* W, float* delta) {
  if (d < 1 || r < 0 || r > d || (r > 0 && (b < 1 || b > 8)) || !U || !lam || !delta || (r > 0 && (!signs || !W)))
    return COBRA_EINVAL;
  if (r == 0) {
    *delta = 0.0f;
    return COBRA_OK;
  }
  std::vector<double> H((size_t)r * r);
  cobra_status st = cobra_hadamard(r, signs, H.data());
  if (st != COBRA_OK) return st;
  // W = U_r H^T: W[i, j] = sum_k U[i, k] H[j, k]
  for (int j = 0; j < r; ++j)
    for (int i = 0; i < d; ++i) {
      double s = 0.0;
      for (int k = 0; k < r; ++k) s += U[(size_t)k * d + i] * H[(size_t)j * r + k];
      W[(size_t)j * d + i] = (float)s;
    }
  double mean = 0.0;
  for (int k = 0; k < r; ++k) mean += lam[k];
  mean /= (double)r;
  double L;
  cobra_loading_factor(b, &L);
  *delta = (float)(2.0 * L * std::sqrt(mean > 0 ? mean : 0.0) / (double)(1 << b));
  return COBRA_OK;
}

// ----------------------------------------------------------------------------------------
// Layout and parameter block.
// ----------------------------------------------------------------------------------------
extern "C" size_t cobra_row_bytes(int r, int b) { return (r > 0 && b > 0) ? (size_t)16 * r * b : 0; }

extern "C" cobra_status cobra_plan_layout(int n_heads, const int* r, const int* b, long long n_slots,
                                          uint64_t* head_offsets, uint64_t* total_bytes) {
  if (n_heads < 0 || n_slots < 0 || (n_heads > 0 && (!r || !b || !head_offsets)) || !total_bytes)
    return COBRA_EINVAL;
  uint64_t pos = 0;
  for (int h = 0; h < n_heads; ++h) {
    if (r[h] < 0 || r[h] > cobra::kD || (r[h] & 1) || (r[h] > 0 && (b[h] < 1 || b[h] > 8))) return COBRA_EINVAL;
    head_offsets[h] = pos;
    pos += (uint64_t)n_slots * cobra_row_bytes(r[h], b[h]);
    pos = align_up(pos, 256);
  }
  *total_bytes = pos;
  return COBRA_OK;
}

namespace {
size_t pool_floats_for(int n_heads, const int* r) {
  size_t f = 0;
  for (int h = 0; h < n_heads; ++h) {
    f = align_up(f, 32) + (size_t)cobra::kD * r[h];
    f = align_up(f, 32) + cobra::kD;
    f = align_up(f, 32) + r[h];
  }
  return align_up(f, 32);
}
}  // namespace

extern "C" cobra_status cobra_params_bytes(int n_heads, const int* r, size_t* bytes) {
  if (n_heads < 1 || !r || !bytes) return COBRA_EINVAL;
  for (int h = 0; h < n_heads; ++h)
    if (r[h] < 0 || r[h] > cobra::kD || (r[h] & 1)) return COBRA_EINVAL;
  const size_t heads_off = sizeof(cobra::BlockHeader);
  const size_t pool_off = align_up(heads_off + sizeof(cobra::HeadEntry) * n_heads, 256);
  *bytes = pool_off + pool_floats_for(n_heads, r) * sizeof(float);
  return COBRA_OK;
}

namespace {
// 64-bit FNV-1a (Fowler-Noll-Vo) over the block, its checksum field taken as zero
uint64_t block_checksum(const unsigned char* p, size_t n) {
  uint64_t h = 14695981039346656037ull;
  const size_t cs = offsetof(cobra::BlockHeader, checksum);
  for (size_t i = 0; i < n; ++i) {
    const unsigned char c = (i >= cs && i < cs + sizeof(uint64_t)) ? 0 : p[i];
    h = (h ^ c) * 1099511628211ull;
  }
  return h;
}

// The block's bytes in host memory (what the device block holds), with its checksum.
cobra_status build_block_image(std::vector<unsigned char>& img, int n_heads, const int* r, const int* b,
                               const float* delta, const uint64_t* cache_off, const float* W_all,
                               const float* mu_all) {
  size_t need = 0;
  cobra_status st = cobra_params_bytes(n_heads, r, &need);
  if (st != COBRA_OK) return st;
  if (!b || !delta || !cache_off || !mu_all) return COBRA_EINVAL;
  size_t total_r = 0;
  for (int h = 0; h < n_heads; ++h) {
    if (r[h] > 0 && (b[h] < 1 || b[h] > 8 || !(delta[h] > 0.0f) || !std::isfinite(delta[h]))) return COBRA_EINVAL;
    if (cache_off[h] & 255) return COBRA_EALIGN;
    total_r += r[h];
  }
  if (total_r > 0 && !W_all) return COBRA_EINVAL;
  img.assign(need, 0);
  auto* hdr = reinterpret_cast<cobra::BlockHeader*>(img.data());
  hdr->magic = cobra::kBlockMagic;
  hdr->version = COBRA_VERSION;
  hdr->n_heads = n_heads;
  hdr->d = cobra::kD;
  hdr->heads_off = sizeof(cobra::BlockHeader);
  hdr->pool_off = align_up(hdr->heads_off + sizeof(cobra::HeadEntry) * n_heads, 256);
  hdr->pool_floats = pool_floats_for(n_heads, r);
  auto* heads = reinterpret_cast<cobra::HeadEntry*>(img.data() + hdr->heads_off);
  float* pool = reinterpret_cast<float*>(img.data() + hdr->pool_off);
  size_t f = 0, wsrc = 0;
  const int d = cobra::kD;
  for (int h = 0; h < n_heads; ++h) {
    cobra::HeadEntry& e = heads[h];
    e.r = r[h];
    e.b = r[h] > 0 ? b[h] : 0;
    e.delta = r[h] > 0 ? delta[h] : 0.0f;
    e.inv_delta = r[h] > 0 ? (float)(1.0 / (double)delta[h]) : 0.0f;
    e.cache_off = cache_off[h];
    f = align_up(f, 32);
    e.w_off = f;
    std::memcpy(pool + f, W_all + wsrc, sizeof(float) * d * r[h]);
    f += (size_t)d * r[h];
    f = align_up(f, 32);
    e.mu_off = f;
    std::memcpy(pool + f, mu_all + (size_t)h * d, sizeof(float) * d);
    f += d;
    f = align_up(f, 32);
    e.wmu_off = f;
    for (int j = 0; j < r[h]; ++j) {
      double s = 0.0;
      for (int i = 0; i < d; ++i) s += (double)W_all[wsrc + (size_t)j * d + i] * (double)mu_all[(size_t)h * d + i];
      pool[f + j] = (float)s;
    }
    f += r[h];
    wsrc += (size_t)d * r[h];
  }
  hdr->checksum = block_checksum(img.data(), img.size());
  return COBRA_OK;
}

cobra_status upload_block(void* dev_block, size_t block_bytes, const void* image, size_t bytes, void* stream) {
  if (!dev_block) return COBRA_EINVAL;
  if (block_bytes < bytes) return COBRA_ESPACE;
  if (((uintptr_t)dev_block) & 255) return COBRA_EALIGN;
  cudaStream_t s = (cudaStream_t)stream;
  if (cudaMemcpyAsync(dev_block, image, bytes, cudaMemcpyHostToDevice, s) != cudaSuccess) return COBRA_ECUDA;
  if (cudaStreamSynchronize(s) != cudaSuccess) return COBRA_ECUDA;
  return COBRA_OK;
}
}  // namespace

extern "C" cobra_status cobra_params_build(void* dev_block, size_t block_bytes, int n_heads, const int* r, const int* b,
                                           const float* delta, const uint64_t* cache_off, const float* W_all,
                                           const float* mu_all, void* stream) {
  size_t need = 0;
  cobra_status st = cobra_params_bytes(n_heads, r, &need);
  if (st != COBRA_OK) return st;
  if (!dev_block || !b || !delta || !cache_off || !mu_all) return COBRA_EINVAL;
  if (block_bytes < need) return COBRA_ESPACE;
  if (((uintptr_t)dev_block) & 255) return COBRA_EALIGN;
  std::vector<unsigned char> img;
  st = build_block_image(img, n_heads, r, b, delta, cache_off, W_all, mu_all);
  if (st != COBRA_OK) return st;
  return upload_block(dev_block, block_bytes, img.data(), img.size(), stream);
}

extern "C" cobra_status cobra_params_image(void* image, size_t image_bytes, int n_heads, const int* r, const int* b,
                                           const float* delta, const uint64_t* cache_off, const float* W_all,
                                           const float* mu_all) {
  size_t need = 0;
  cobra_status st = cobra_params_bytes(n_heads, r, &need);
  if (st != COBRA_OK) return st;
  if (!image) return COBRA_EINVAL;
  if (image_bytes < need) return COBRA_ESPACE;
  std::vector<unsigned char> img;
  st = build_block_image(img, n_heads, r, b, delta, cache_off, W_all, mu_all);
  if (st != COBRA_OK) return st;
  std::memcpy(image, img.data(), img.size());
  return COBRA_OK;
}

extern "C" cobra_status cobra_params_verify(const void* image, size_t image_bytes) {
  if (!image || image_bytes < sizeof(cobra::BlockHeader)) return COBRA_EINVAL;
  const auto* p = static_cast<const unsigned char*>(image);
  cobra::BlockHeader hdr;
  std::memcpy(&hdr, p, sizeof(hdr));
  if (hdr.magic != cobra::kBlockMagic || hdr.version != COBRA_VERSION || hdr.d != cobra::kD || hdr.n_heads < 1 ||
      hdr.n_heads > (1 << 20) || hdr.heads_off != sizeof(cobra::BlockHeader))
    return COBRA_EINVAL;
  const size_t n = (size_t)hdr.n_heads;
  if (hdr.pool_off != align_up(hdr.heads_off + sizeof(cobra::HeadEntry) * n, 256) || hdr.pool_off > image_bytes)
    return COBRA_EINVAL;
  std::vector<int> r(n);
  for (size_t h = 0; h < n; ++h) {
    cobra::HeadEntry e;
    std::memcpy(&e, p + hdr.heads_off + h * sizeof(e), sizeof(e));
    r[h] = e.r;
    if (e.r < 0 || e.r > cobra::kD || (e.r & 1)) return COBRA_EINVAL;
  }
  size_t need = 0;
  if (cobra_params_bytes((int)n, r.data(), &need) != COBRA_OK || need != image_bytes ||
      hdr.pool_floats != pool_floats_for((int)n, r.data()))
    return COBRA_EINVAL;
  for (size_t h = 0; h < n; ++h) {
    cobra::HeadEntry e;
    std::memcpy(&e, p + hdr.heads_off + h * sizeof(e), sizeof(e));
    // the same head fields cobra_params_build writes: for r > 0 a finite positive step and its
    // reciprocal rounded from double, bit for bit; for r = 0 zeros
    if (e.r > 0) {
      if (e.b < 1 || e.b > 8 || !(e.delta > 0.0f) || !std::isfinite(e.delta)) return COBRA_EINVAL;
      const float inv = (float)(1.0 / (double)e.delta);
      if (std::memcmp(&inv, &e.inv_delta, sizeof(float)) != 0) return COBRA_EINVAL;
    } else if (e.b != 0 || e.delta != 0.0f || e.inv_delta != 0.0f) {
      return COBRA_EINVAL;
    }
    if (e.w_off + (uint64_t)cobra::kD * e.r > hdr.pool_floats || e.mu_off + cobra::kD > hdr.pool_floats ||
        e.wmu_off + (uint64_t)e.r > hdr.pool_floats || (e.cache_off & 255))
      return COBRA_EINVAL;
  }
  return block_checksum(p, image_bytes) == hdr.checksum ? COBRA_OK : COBRA_EINVAL;
}

extern "C" cobra_status cobra_params_upload(void* dev_block, size_t block_bytes, const void* image, size_t image_bytes,
                                            void* stream) {
  const cobra_status st = cobra_params_verify(image, image_bytes);
  if (st != COBRA_OK) return st;
  return upload_block(dev_block, block_bytes, image, image_bytes, stream);
}

// ----------------------------------------------------------------------------------------
// Decode work plan: per (seq, layer, kv-head) group, token chunks of whole code rows.  The
// scan's warps take the chunks in plan order, and the chunk sizes shrink towards the end of
// the list (guided self-scheduling): a chunk holds about the packed K+V bytes still ahead of it
// divided by kGuide x kScanWarps, clamped to [kItemMin, kItemMax], and no group is cut into
// more than about kMaxChunks chunks (the combine merges a group's chunks).  Most of the cache
// goes in large chunks (little per-chunk setup), and the warps that drain the queue finish
// within one short chunk of one another.  Groups are ordered by code variant (b_K, b_V), then
// (r_K, r_V), so that the warps working at the same time run the same code.
// ----------------------------------------------------------------------------------------
namespace {
constexpr long long kItemMin = 16 * 1024, kItemMax = 128 * 1024;
constexpr long long kScanWarps = 152 * 16;  // resident scan warps: 152 SMs x 4 CTAs x 4 warps
constexpr long long kGuide = 2;
constexpr long long kMaxChunks = 32;

cobra_status check_decode_desc(const cobra_decode_desc* d) {
  if (!d) return COBRA_EINVAL;
  if (d->n_layers < 1 || d->n_kv_heads < 1 || d->n_seqs < 1 || (d->group != 4 && d->group != 8) ||
      d->layer_stride < d->n_kv_heads || d->k_head0 < 0 || d->v_head0 < 0)
    return COBRA_EINVAL;
  return COBRA_OK;
}

struct Plan {
  std::vector<cobra::WsGroup> groups;
  std::vector<cobra::WsItem> items;
  int max_rv = 0, max_row_bytes = 0;
  int max_stage_bytes = 0;  // largest K channel tiles + V row (128-byte aligned) of a group
};

cobra_status make_plan(const cobra_decode_desc* d, const int* head_r, const int* head_b, const int* seq_cap, Plan& p) {
  cobra_status st = check_decode_desc(d);
  if (st != COBRA_OK) return st;
  if (!head_r || !head_b || !seq_cap) return COBRA_EINVAL;
  for (int s = 0; s < d->n_seqs; ++s) {
    if (seq_cap[s] < 0) return COBRA_EINVAL;
    long long rows = (seq_cap[s] + 127) / 128;
    if (rows > 65535) return COBRA_EINVAL;
    if (!d->pages_per_seq && rows > d->rows_per_seq) return COBRA_EINVAL;
    if (d->pages_per_seq && rows > 2LL * d->pages_per_seq) return COBRA_EINVAL;
  }
  struct Key {
    int bk, bv, rk, rv, s, l, h;
  };
  std::vector<Key> keys;
  for (int s = 0; s < d->n_seqs; ++s)
    for (int l = 0; l < d->n_layers; ++l)
      for (int h = 0; h < d->n_kv_heads; ++h) {
        const int hk = d->k_head0 + l * d->layer_stride + h, hv = d->v_head0 + l * d->layer_stride + h;
        const int rk = head_r[hk], rv = head_r[hv], bk = rk ? head_b[hk] : 0, bv = rv ? head_b[hv] : 0;
        if (rk < 0 || rk > 128 || (rk & 1) || rv < 0 || rv > 128 || (rv & 1) || bk < 0 || bk > 8 || bv < 0 || bv > 8)
          return COBRA_EINVAL;
        keys.push_back({bk, bv, rk, rv, s, l, h});
      }
  std::stable_sort(keys.begin(), keys.end(), [](const Key& x, const Key& y) {
    if (x.bk != y.bk) return x.bk < y.bk;
    if (x.bv != y.bv) return x.bv < y.bv;
    if (x.rk != y.rk) return x.rk < y.rk;
    return x.rv < y.rv;
  });
  auto pair_bytes = [](const Key& k) {
    return (long long)cobra_row_bytes(k.rk, k.bk) + (long long)cobra_row_bytes(k.rv, k.bv);
  };
  long long remaining = 0;  // packed K+V bytes not yet in a chunk
  for (const Key& k : keys) remaining += (long long)(seq_cap[k.s] + 127) / 128 * pair_bytes(k);
  for (const Key& key : keys) {
    const int hk = d->k_head0 + key.l * d->layer_stride + key.h, hv = d->v_head0 + key.l * d->layer_stride + key.h;
    p.max_rv = std::max(p.max_rv, key.rv);
    p.max_row_bytes =
        std::max(p.max_row_bytes, (int)std::max(cobra_row_bytes(key.rk, key.bk), cobra_row_bytes(key.rv, key.bv)));
    p.max_stage_bytes = std::max(p.max_stage_bytes, 256 * key.bk * ((key.rk + 15) / 16) +
                                                        (int)align_up(cobra_row_bytes(key.rv, key.bv), 128));
    const long long rows = (seq_cap[key.s] + 127) / 128, rb = pair_bytes(key);
    cobra::WsGroup g{key.s, key.l, key.h, (int)p.items.size(), 0, hk, hv, 0};
    if (rows == 0 || rb == 0) {  // one (empty or code-less) chunk
      p.items.push_back({(int)p.groups.size(), 0, (int)rows, (int)p.items.size()});
      g.n_items = 1;
    }
    const long long min_rows = (rows + kMaxChunks - 1) / kMaxChunks;
    for (long long r0 = 0; r0 < rows && rb > 0;) {
      const long long target = std::min(kItemMax, std::max(kItemMin, remaining / (kGuide * kScanWarps)));
      long long n = std::max(min_rows, std::max(1LL, (target + rb / 2) / rb));
      if (rows - r0 - n < (n + 1) / 2) n = rows - r0;  // no short remainder chunk
      p.items.push_back({(int)p.groups.size(), (int)r0, (int)(r0 + n), (int)p.items.size()});
      g.n_items++;
      r0 += n;
      remaining -= n * rb;
    }
    p.groups.push_back(g);
  }
  return COBRA_OK;
}

void ws_layout(const cobra_decode_desc* d, const Plan& p, cobra::WsHeader& h, size_t& bytes) {
  std::memset(&h, 0, sizeof(h));
  h.magic = cobra::kWsMagic;
  h.version = COBRA_VERSION;
  h.n_groups = (int)p.groups.size();
  h.n_items = (int)p.items.size();
  h.group = d->group;
  h.n_layers = d->n_layers;
  h.n_kv = d->n_kv_heads;
  h.n_seqs = d->n_seqs;
  h.max_rv = p.max_rv;
  h.max_row_bytes = p.max_row_bytes;
  h.g_stride = 4 + (int)align_up((size_t)p.max_rv, 4);
  h.part_stride = h.g_stride * d->group;
  h.qt_stride = cobra::kQtStride;
  size_t off = sizeof(cobra::WsHeader);
  h.groups_off = off = align_up(off, 256);
  off += sizeof(cobra::WsGroup) * p.groups.size();
  h.items_off = off = align_up(off, 256);
  off += sizeof(cobra::WsItem) * p.items.size();
  h.hg_off = off = align_up(off, 256);
  off += sizeof(int32_t) * p.groups.size();
  h.qt_off = off = align_up(off, 256);
  off += (size_t)h.qt_stride * p.groups.size();
  h.part_off = off = align_up(off, 256);
  off += sizeof(float) * (size_t)h.part_stride * p.items.size();
  bytes = align_up(off, 256);
}
}  // namespace

extern "C" cobra_status cobra_decode_workspace_size(const cobra_decode_desc* desc, const int* head_r,
                                                    const int* head_b, const int* seq_cap, size_t* bytes) {
  if (!bytes) return COBRA_EINVAL;
  Plan p;
  cobra_status st = make_plan(desc, head_r, head_b, seq_cap, p);
  if (st != COBRA_OK) return st;
  cobra::WsHeader h;
  ws_layout(desc, p, h, *bytes);
  return COBRA_OK;
}

namespace {
// header + groups + items + head-group table of the workspace, as a host image
cobra_status plan_image(const cobra_decode_desc* desc, const int* head_r, const int* head_b, const int* seq_cap,
                        std::vector<unsigned char>& img, size_t* ws_need, cobra_decode_info* info) {
  Plan p;
  cobra_status st = make_plan(desc, head_r, head_b, seq_cap, p);
  if (st != COBRA_OK) return st;
  cobra::WsHeader h;
  ws_layout(desc, p, h, *ws_need);
  const size_t head_bytes = h.qt_off;
  img.assign(head_bytes, 0);
  std::memcpy(img.data(), &h, sizeof(h));
  std::memcpy(img.data() + h.groups_off, p.groups.data(), sizeof(cobra::WsGroup) * p.groups.size());
  std::memcpy(img.data() + h.items_off, p.items.data(), sizeof(cobra::WsItem) * p.items.size());
  int32_t* hg = reinterpret_cast<int32_t*>(img.data() + h.hg_off);
  for (size_t g = 0; g < p.groups.size(); ++g) {
    const cobra::WsGroup& gr = p.groups[g];
    hg[((size_t)gr.layer * desc->n_kv_heads + gr.kv) * desc->n_seqs + gr.seq] = (int32_t)g;
  }
  info->n_groups = h.n_groups;
  info->n_items = h.n_items;
  info->max_row_bytes = h.max_row_bytes;
  info->max_stage_bytes = p.max_stage_bytes;
  return COBRA_OK;
}
}  // namespace

extern "C" cobra_status cobra_decode_plan_host(const cobra_decode_desc* desc, const int* head_r, const int* head_b,
                                               const int* seq_cap, void* image, size_t image_bytes, size_t* written,
                                               cobra_decode_info* info) {
  if (!written || !info) return COBRA_EINVAL;
  std::vector<unsigned char> img;
  size_t need = 0;
  cobra_decode_info inf{};
  cobra_status st = plan_image(desc, head_r, head_b, seq_cap, img, &need, &inf);
  if (st != COBRA_OK) return st;
  *written = img.size();
  if (!image) return COBRA_EINVAL;
  if (image_bytes < img.size()) return COBRA_ESPACE;
  std::memcpy(image, img.data(), img.size());
  *info = inf;
  return COBRA_OK;
}

extern "C" cobra_status cobra_decode_plan(const cobra_decode_desc* desc, const int* head_r, const int* head_b,
                                          const int* seq_cap, void* workspace, size_t ws_bytes, cobra_decode_info* info,
                                          void* stream) {
  if (!workspace || !info) return COBRA_EINVAL;
  if (((uintptr_t)workspace) & 255) return COBRA_EALIGN;
  std::vector<unsigned char> img;
  size_t need = 0;
  cobra_decode_info inf{};
  cobra_status st = plan_image(desc, head_r, head_b, seq_cap, img, &need, &inf);
  if (st != COBRA_OK) return st;
  if (ws_bytes < need) return COBRA_ESPACE;
  cudaStream_t s = (cudaStream_t)stream;
  if (cudaMemcpyAsync(workspace, img.data(), img.size(), cudaMemcpyHostToDevice, s) != cudaSuccess) return COBRA_ECUDA;
  if (cudaStreamSynchronize(s) != cudaSuccess) return COBRA_ECUDA;
  *info = inf;
  return COBRA_OK;
}
