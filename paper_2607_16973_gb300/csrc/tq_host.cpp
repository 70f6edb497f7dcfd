// Host-side parts of the C ABI: error plumbing, thread-local settings, the
// Lloyd-Max codebook (Sec. II-B step 3) and the random rotation (Sec. II-B
// step 2).  Pure C++ (no CUDA), OpenMP for the rotation's column updates.
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <exception>
#include <new>
#include <string>
#include <vector>

#include <omp.h>

#include "tq_internal.h"

namespace tq {

namespace {
thread_local std::string g_error;
thread_local int g_path = TQ_PATH_AUTO;
thread_local void* g_prof_start = nullptr;
thread_local void* g_prof_stop = nullptr;
}  // namespace

tq_status fail(tq_status st, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  g_error = buf;
  return st;
}

tq_status ok() {
  g_error.clear();
  return TQ_OK;
}

int search_path() { return g_path; }
void* profile_start() { return g_prof_start; }
void* profile_stop() { return g_prof_stop; }

// ---------------------------------------------------------------------------
// Codebook: Lloyd-Max on the analytic coordinate marginal.
//
// Moments over a cell are integrated with composite 16-point Gauss-Legendre
// on panels no wider than sigma/4 (sigma = 1/sqrt(d), the marginal's standard
// deviation), clipped to the support: [-1, 1] for the Beta marginal, and
// +-40 sigma for the Gaussian (beyond which the density underflows a double).
// The Lloyd-Max conditions c_i = E[x | t_{i-1} < x <= t_i], t_i = (c_i +
// c_{i+1})/2 are solved by a few Lloyd steps followed by Newton's method on
// T(c) - c = 0, whose Jacobian is tridiagonal:
//   dT_i/dt_i     = f(t_i) (t_i - T_i) / M0_i,
//   dT_i/dt_{i-1} = f(t_{i-1}) (T_i - t_{i-1}) / M0_i,   dt_i/dc = 1/2.
// ---------------------------------------------------------------------------
namespace {

struct GaussLegendre16 {
  double x[16], w[16];
  GaussLegendre16() {
    const int n = 16;
    for (int i = 0; i < n; ++i) {
      // Newton on P_n starting from the Chebyshev-like guess.
      double z = std::cos(M_PI * (i + 0.75) / (n + 0.5));
      for (int it = 0; it < 100; ++it) {
        double p0 = 1.0, p1 = z;
        for (int k = 2; k <= n; ++k) {
          double p2 = ((2.0 * k - 1.0) * z * p1 - (k - 1.0) * p0) / k;
          p0 = p1;
          p1 = p2;
        }
        double dp = n * (z * p1 - p0) / (z * z - 1.0);
        double dz = p1 / dp;
        z -= dz;
        if (std::fabs(dz) < 1e-16) {
          // recompute the derivative at the converged node for the weight
          p0 = 1.0;
          p1 = z;
          for (int k = 2; k <= n; ++k) {
            double p2 = ((2.0 * k - 1.0) * z * p1 - (k - 1.0) * p0) / k;
            p0 = p1;
            p1 = p2;
          }
          dp = n * (z * p1 - p0) / (z * z - 1.0);
          x[i] = z;
          w[i] = 2.0 / ((1.0 - z * z) * dp * dp);
          break;
        }
      }
    }
  }
};

const GaussLegendre16& gl16() {
  static const GaussLegendre16 g;
  return g;
}

struct Marginal {
  int d;
  int kind;
  double m, logc, sigma, lo, hi;
  Marginal(int d_, int kind_) : d(d_), kind(kind_) {
    sigma = 1.0 / std::sqrt((double)d);
    if (kind == TQ_MARGINAL_BETA) {
      m = 0.5 * (d - 3);
      logc = std::lgamma(0.5 * d) - std::lgamma(0.5 * (d - 1)) - 0.5 * std::log(M_PI);
      lo = -1.0;
      hi = 1.0;
    } else {
      m = 0.0;
      logc = -std::log(sigma * std::sqrt(2.0 * M_PI));
      lo = -40.0 * sigma;
      hi = 40.0 * sigma;
    }
  }
  double pdf(double x) const {
    if (x <= lo || x >= hi) return 0.0;
    if (kind == TQ_MARGINAL_BETA) return std::exp(logc + m * std::log1p(-x * x));
    double z = x / sigma;
    return std::exp(logc - 0.5 * z * z);
  }
  // int_a^b x^p f(x) dx for p = 0, 1, 2 (and (x - c)^2 f when c is given)
  void moments(double a, double b, double c, double out[4]) const {
    out[0] = out[1] = out[2] = out[3] = 0.0;
    a = std::max(a, lo);
    b = std::min(b, hi);
    if (!(b > a)) return;
    const GaussLegendre16& g = gl16();
    const double h = 0.25 * sigma;
    const int panels = std::max(1, (int)std::ceil((b - a) / h));
    const double w = (b - a) / panels;
    for (int p = 0; p < panels; ++p) {
      const double pa = a + p * w;
      const double mid = pa + 0.5 * w, half = 0.5 * w;
      for (int i = 0; i < 16; ++i) {
        const double x = mid + half * g.x[i];
        const double fx = pdf(x) * g.w[i] * half;
        out[0] += fx;
        out[1] += fx * x;
        out[2] += fx * x * x;
        out[3] += fx * (x - c) * (x - c);
      }
    }
  }
};

// Quantiles (i + 1/2)/L of the marginal, from the cumulative integral on a
// fine grid, used as the starting centroids.
std::vector<double> quantile_init(const Marginal& f, int L) {
  const int G = 20000;
  const double a = std::max(f.lo, -12.0 * f.sigma), b = std::min(f.hi, 12.0 * f.sigma);
  std::vector<double> xs(G + 1), cdf(G + 1, 0.0);
  for (int i = 0; i <= G; ++i) xs[i] = a + (b - a) * i / G;
  for (int i = 0; i < G; ++i) {
    double mo[4];
    f.moments(xs[i], xs[i + 1], 0.0, mo);
    cdf[i + 1] = cdf[i] + mo[0];
  }
  std::vector<double> c(L);
  for (int i = 0; i < L; ++i) {
    const double p = (i + 0.5) / L * cdf[G];
    int j = (int)(std::lower_bound(cdf.begin(), cdf.end(), p) - cdf.begin());
    j = std::min(std::max(j, 1), G);
    const double span = cdf[j] - cdf[j - 1];
    const double frac = span > 0 ? (p - cdf[j - 1]) / span : 0.5;
    c[i] = xs[j - 1] + frac * (xs[j] - xs[j - 1]);
  }
  return c;
}

void lloyd_map(const Marginal& f, const std::vector<double>& c, std::vector<double>& t,
               std::vector<double>& T, std::vector<double>& M0) {
  const int L = (int)c.size();
  t.resize(L + 1);
  t[0] = f.lo;
  t[L] = f.hi;
  for (int i = 1; i < L; ++i) t[i] = 0.5 * (c[i - 1] + c[i]);
  T.resize(L);
  M0.resize(L);
  for (int i = 0; i < L; ++i) {
    double mo[4];
    f.moments(t[i], t[i + 1], 0.0, mo);
    M0[i] = mo[0];
    T[i] = mo[0] > 0 ? mo[1] / mo[0] : 0.5 * (t[i] + t[i + 1]);
  }
}

bool increasing(const std::vector<double>& c, double lo, double hi) {
  for (size_t i = 0; i < c.size(); ++i) {
    if (!(c[i] > lo && c[i] < hi)) return false;
    if (i && !(c[i] > c[i - 1])) return false;
  }
  return true;
}

std::vector<double> solve_lloyd_max(const Marginal& f, int L) {
  std::vector<double> c = quantile_init(f, L), t, T, M0;
  for (int it = 0; it < 40; ++it) {  // a few plain Lloyd steps
    lloyd_map(f, c, t, T, M0);
    c = T;
  }
  const double scale = std::fabs(c.back());
  for (int it = 0; it < 200; ++it) {
    lloyd_map(f, c, t, T, M0);
    // (I - J) delta = T - c with J the tridiagonal Jacobian of the Lloyd map
    std::vector<double> lower(L, 0.0), diag(L, 1.0), upper(L, 0.0), rhs(L);
    for (int i = 0; i < L; ++i) {
      rhs[i] = T[i] - c[i];
      if (M0[i] <= 0) continue;
      const double jl = (i > 0) ? 0.5 * f.pdf(t[i]) * (T[i] - t[i]) / M0[i] : 0.0;
      const double ju = (i < L - 1) ? 0.5 * f.pdf(t[i + 1]) * (t[i + 1] - T[i]) / M0[i] : 0.0;
      lower[i] = -jl;
      upper[i] = -ju;
      diag[i] = 1.0 - jl - ju;
    }
    // Thomas algorithm
    for (int i = 1; i < L; ++i) {
      const double w = lower[i] / diag[i - 1];
      diag[i] -= w * upper[i - 1];
      rhs[i] -= w * rhs[i - 1];
    }
    std::vector<double> delta(L);
    delta[L - 1] = rhs[L - 1] / diag[L - 1];
    for (int i = L - 2; i >= 0; --i) delta[i] = (rhs[i] - upper[i] * delta[i + 1]) / diag[i];
    std::vector<double> cn(L);
    double move = 0.0;
    for (int i = 0; i < L; ++i) {
      cn[i] = c[i] + delta[i];
      move = std::max(move, std::fabs(delta[i]));
    }
    if (!increasing(cn, f.lo, f.hi)) {
      c = T;  // fall back to a Lloyd step
      continue;
    }
    c = cn;
    if (move <= 1e-15 * scale) break;
  }
  // the fixed point of a symmetric log-concave marginal is symmetric
  std::vector<double> s(L);
  for (int i = 0; i < L; ++i) s[i] = 0.5 * (c[i] - c[L - 1 - i]);
  return s;
}

}  // namespace
}  // namespace tq

extern "C" const char* tq_last_error(void) { return tq::g_error.c_str(); }

extern "C" int tq_version(void) { return 100; }

extern "C" tq_status tq_set_search_path(int path) {
  if (path != TQ_PATH_AUTO && path != TQ_PATH_LUT && path != TQ_PATH_MMA && path != TQ_PATH_LUT_FIXED &&
      path != TQ_PATH_LUT_FOLD)
    return tq::fail(TQ_EINVAL, "tq_set_search_path: unknown path %d", path);
  tq::g_path = path;
  return tq::ok();
}

extern "C" tq_status tq_profile_events(void* scan_start, void* scan_stop) {
  if ((scan_start == nullptr) != (scan_stop == nullptr))
    return tq::fail(TQ_EINVAL, "tq_profile_events: give both events or neither");
  tq::g_prof_start = scan_start;
  tq::g_prof_stop = scan_stop;
  return tq::ok();
}

extern "C" tq_status tq_codebook(int d, int bits, int marginal, float* centroids,
                                 float* boundaries, double* distortion) {
  try {
    if (d < 8 || d > 1 << 24) return tq::fail(TQ_EINVAL, "tq_codebook: d=%d outside [8, 2^24]", d);
    if (bits < 1 || bits > 8) return tq::fail(TQ_EINVAL, "tq_codebook: bits=%d outside [1, 8]", bits);
    if (marginal != TQ_MARGINAL_BETA && marginal != TQ_MARGINAL_GAUSS)
      return tq::fail(TQ_EINVAL, "tq_codebook: unknown marginal %d", marginal);
    if (!centroids || !boundaries) return tq::fail(TQ_EINVAL, "tq_codebook: NULL output");
    const int L = 1 << bits;
    tq::Marginal f(d, marginal);
    std::vector<double> c = tq::solve_lloyd_max(f, L);
    double D = 0.0;
    for (int i = 0; i < L; ++i) {
      const double a = i ? 0.5 * (c[i - 1] + c[i]) : f.lo;
      const double b = i < L - 1 ? 0.5 * (c[i] + c[i + 1]) : f.hi;
      double mo[4];
      f.moments(a, b, c[i], mo);
      D += mo[3];
      centroids[i] = (float)c[i];
      if (i < L - 1) boundaries[i] = (float)(0.5 * (c[i] + c[i + 1]));
    }
    if (distortion) *distortion = D;
    return tq::ok();
  } catch (const std::bad_alloc&) {
    return tq::fail(TQ_ENOMEM, "tq_codebook: out of host memory");
  } catch (const std::exception& e) {
    return tq::fail(TQ_EINVAL, "tq_codebook: %s", e.what());
  }
}

// ---------------------------------------------------------------------------
// Rotation: splitmix64 -> Box-Muller -> Householder QR -> Q diag(sign(diag U)).
// ---------------------------------------------------------------------------
namespace tq {
namespace {

// y -= (beta * <x, y>) x over len entries; eight partial sums so the dot
// product vectorises.
inline void apply_reflector(const double* x, double* y, int64_t len, double beta) {
  double acc[8] = {0, 0, 0, 0, 0, 0, 0, 0};
  int64_t i = 0;
  for (; i + 8 <= len; i += 8)
    for (int u = 0; u < 8; ++u) acc[u] += x[i + u] * y[i + u];
  for (; i < len; ++i) acc[0] += x[i] * y[i];
  const double w = beta * (((acc[0] + acc[1]) + (acc[2] + acc[3])) + ((acc[4] + acc[5]) + (acc[6] + acc[7])));
  for (int64_t j = 0; j < len; ++j) y[j] -= w * x[j];
}

// Thread count for the rotation: one core is left free, because the
// reflector loop has ~2d short parallel regions and a thread that loses its
// core stalls every barrier.
inline int rotation_threads() {
  return std::max(1, std::min(omp_get_num_procs() - 1, omp_get_max_threads()));
}

inline uint64_t splitmix64_at(uint64_t seed, uint64_t counter) {
  uint64_t z = seed + (counter + 1) * 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

}  // namespace
}  // namespace tq

extern "C" tq_status tq_rotation(int d, uint64_t seed, float* R) {
  try {
    if (d < 2 || d > tq::kMaxD) return tq::fail(TQ_EINVAL, "tq_rotation: d=%d outside [2, %d]", d, tq::kMaxD);
    if (!R) return tq::fail(TQ_EINVAL, "tq_rotation: NULL output");
    const int64_t D = d;
    // A: column-major d x d, A[j*d + i] = G(i, j); G is filled row-major.
    std::vector<double> A(D * D);
    const int64_t total = D * D, pairs = (total + 1) / 2;
    const int nth = tq::rotation_threads();
#pragma omp parallel for schedule(static) num_threads(nth)
    for (int64_t p = 0; p < pairs; ++p) {
      const uint64_t a = tq::splitmix64_at(seed, 2 * (uint64_t)p);
      const uint64_t b = tq::splitmix64_at(seed, 2 * (uint64_t)p + 1);
      const double u1 = ((double)(a >> 11) + 1.0) * 0x1p-53;
      const double u2 = (double)(b >> 11) * 0x1p-53;
      const double r = std::sqrt(-2.0 * std::log(u1));
      const double th = 2.0 * M_PI * u2;
      const int64_t e0 = 2 * p, e1 = 2 * p + 1;
      A[(e0 % D) * D + e0 / D] = r * std::cos(th);
      if (e1 < total) A[(e1 % D) * D + e1 / D] = r * std::sin(th);
    }
    // Householder QR: column k's reflector v_k (stored in A[k.., k]) maps
    // A[k.., k] to diag[k] e_0.
    std::vector<double> diag(D), vtv(D);
    for (int64_t k = 0; k < D; ++k) {
      double* x = &A[k * D + k];
      const int64_t len = D - k;
      double nrm2 = 0.0;
      for (int64_t i = 0; i < len; ++i) nrm2 += x[i] * x[i];
      const double alpha = std::sqrt(nrm2);
      if (alpha == 0.0) {
        diag[k] = 0.0;
        vtv[k] = 0.0;
        continue;
      }
      const double s = x[0] >= 0 ? 1.0 : -1.0;
      diag[k] = -s * alpha;
      x[0] += s * alpha;
      vtv[k] = 2.0 * alpha * (alpha + std::fabs(x[0] - s * alpha));
      const double beta = 2.0 / vtv[k];
#pragma omp parallel for schedule(dynamic, 16) num_threads(nth) if (len * (D - k) > 65536)
      for (int64_t j = k + 1; j < D; ++j) tq::apply_reflector(x, &A[j * D + k], len, beta);
    }
    // Q = H_0 H_1 ... H_{d-1}, accumulated backwards into Qm (column-major).
    std::vector<double> Qm(D * D, 0.0);
    for (int64_t i = 0; i < D; ++i) Qm[i * D + i] = 1.0;
    for (int64_t k = D - 1; k >= 0; --k) {
      if (vtv[k] == 0.0) continue;
      const double* x = &A[k * D + k];
      const int64_t len = D - k;
      const double beta = 2.0 / vtv[k];
#pragma omp parallel for schedule(dynamic, 16) num_threads(nth) if (len * (D - k) > 65536)
      for (int64_t j = k; j < D; ++j) tq::apply_reflector(x, &Qm[j * D + k], len, beta);
    }
    // sign fix: G = (Q S)(S U) with S = diag(sign U_kk) gives a positive diagonal
    for (int64_t j = 0; j < D; ++j) {
      const double sgn = diag[j] < 0 ? -1.0 : 1.0;
      for (int64_t i = 0; i < D; ++i) R[i * D + j] = (float)(sgn * Qm[j * D + i]);
    }
    return tq::ok();
  } catch (const std::bad_alloc&) {
    return tq::fail(TQ_ENOMEM, "tq_rotation: out of host memory");
  } catch (const std::exception& e) {
    return tq::fail(TQ_EINVAL, "tq_rotation: %s", e.what());
  }
}
