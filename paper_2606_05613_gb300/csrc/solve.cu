// Solve pass: one warp per bucket.
//
// The warp first reduces the bucket's per-chunk Gram partials in a fixed
// order (lane p owns entry p of the triangle and adds the chunks in
// ascending order, in fp64), giving the bucket's K x K Gram matrix G in
// shared memory.  Lane 0 then solves the bucket's rule on G in fp64 and
// writes the coefficients beta (d_b = sum_k beta_k g_k):
//
//  MGDA (Eq. 3; bucket form Eq. 6 over the simplex of Algorithm 1):
//    K = 2: gamma = clamp(<g2 - g1, g2> / ||g1 - g2||^2, 0, 1).
//    Otherwise Frank-Wolfe from the best pair with exact line search, then
//    (POLISH) an exact active-set completion in the manner of Wolfe's
//    minimum-norm-point algorithm: the affine minimum-norm point of the
//    current support is taken when it lies inside the simplex, else the
//    iterate moves to the boundary and drops a point; a point is added while
//    some g_j has <d, g_j> < ||d||^2.
//  CAGrad (Eq. 4; Eq. 7): the dual min_{w in simplex} F(w),
//    F(w) = <g0, g_w> + c ||g0|| ||g_w||, by Frank-Wolfe with exact line
//    search from the best vertex, then (POLISH) the same kind of active-set
//    completion with the closed-form stationary point of F on the affine
//    hull of the support; beta = 1/K + c ||g0|| w / ||g_w||.
//  PCGrad (Eq. 5; Eq. 8): the projections of Algorithm 1 carried out on the
//    coefficients of each running d_t, since <d_t, g_j> = sum_m C_tm G_mj.
//  MEAN: beta = 1/K.
//
// All solvers work on G scaled so that max_k G_kk = 1 (every rule is
// invariant under a positive scaling of G).  A Gram with a NaN or Inf gives
// beta = 1/K and status BKMOO_ERR_NONFINITE.
#include <math.h>

#include "common.cuh"

namespace bkmoo {
namespace {

constexpr double kInside = 1e-15;  // weights above this are in the support
constexpr double kKkt = 1e-13;     // optimality slack on the normalised Gram
constexpr double kPivot = 1e-13;   // smallest pivot of a non-singular system

// ---------------------------------------------------------------------------
// partial reduction
// ---------------------------------------------------------------------------

__device__ void reduce_bucket(const PlanView& v, int64_t b, double* G, int lane) {
  const int K = v.K, P = tri(K);
  const int64_t c0 = v.chunk_prefix[b], c1 = v.chunk_prefix[b + 1];
  for (int p = lane; p < P; p += 32) {
    double s = 0.0;
    const double* src = v.partials + c0 * P + p;
    for (int64_t c = c0; c < c1; ++c, src += P) s += *src;
    int i = 0, r = p;
    while (r >= K - i) {
      r -= K - i;
      ++i;
    }
    const int j = i + r;
    G[i * K + j] = s;
    G[j * K + i] = s;
  }
  __syncwarp();
}

// ---------------------------------------------------------------------------
// small dense helpers (lane 0 only)
// ---------------------------------------------------------------------------

__device__ void mat_vec(int K, const double* G, const double* x, double* y) {
  for (int i = 0; i < K; ++i) {
    double s = 0.0;
    for (int j = 0; j < K; ++j) s += G[i * K + j] * x[j];
    y[i] = s;
  }
}

__device__ double dotk(int K, const double* a, const double* c) {
  double s = 0.0;
  for (int k = 0; k < K; ++k) s += a[k] * c[k];
  return s;
}

__device__ int argmin_first(int K, const double* v) {
  int t = 0;
  for (int k = 1; k < K; ++k)
    if (v[k] < v[t]) t = k;
  return t;
}

// In-place Gauss-Jordan elimination with partial pivoting of an m x (m + r)
// augmented matrix (row stride m + r); the r solution columns end up in
// columns m .. m + r - 1.  False when a pivot is below kPivot.
__device__ bool gauss_jordan(double* A, int m, int r) {
  const int n = m + r;
  for (int c = 0; c < m; ++c) {
    int piv = c;
    double big = fabs(A[c * n + c]);
    for (int i = c + 1; i < m; ++i) {
      const double t = fabs(A[i * n + c]);
      if (t > big) {
        big = t;
        piv = i;
      }
    }
    if (!(big > kPivot)) return false;
    if (piv != c)
      for (int j = 0; j < n; ++j) {
        const double t = A[c * n + j];
        A[c * n + j] = A[piv * n + j];
        A[piv * n + j] = t;
      }
    const double inv = 1.0 / A[c * n + c];
    for (int j = c; j < n; ++j) A[c * n + j] *= inv;
    for (int i = 0; i < m; ++i) {
      if (i == c) continue;
      const double f = A[i * n + c];
      if (f == 0.0) continue;
      for (int j = c; j < n; ++j) A[i * n + j] -= f * A[c * n + j];
    }
  }
  return true;
}

// Minimiser of ||sum_{i<s} y_i g_{S_i}||^2 with sum y = 1 (sign free): the
// bordered stationarity system [G_SS 1; 1^T 0].
__device__ bool affine_min_norm(int K, const double* G, const int* S, int s, double* y) {
  double A[(kMaxK + 1) * (kMaxK + 2)];
  const int m = s + 1, n = m + 1;
  for (int i = 0; i < s; ++i) {
    for (int j = 0; j < s; ++j) A[i * n + j] = G[S[i] * K + S[j]];
    A[i * n + s] = 1.0;
    A[i * n + m] = 0.0;
  }
  for (int j = 0; j < s; ++j) A[s * n + j] = 1.0;
  A[s * n + s] = 0.0;
  A[s * n + m] = 1.0;
  if (!gauss_jordan(A, m, 1)) return false;
  for (int i = 0; i < s; ++i) y[i] = A[i * n + m];
  return true;
}

// Move w (supported on S) towards y (affine point of S, some y_i <= kInside)
// up to the boundary of the simplex and drop the support points whose weight
// reaches 0.  Returns the new support size.
__device__ int step_to_boundary(double* w, int* S, int s, const double* y) {
  double theta = 1.0;
  int drop = -1;
  for (int i = 0; i < s; ++i) {
    if (y[i] > kInside) continue;
    const double a = w[S[i]], den = a - y[i];
    const double t = den > 0.0 ? a / den : 0.0;
    if (drop < 0 || t < theta) {
      theta = t;
      drop = i;
    }
  }
  for (int i = 0; i < s; ++i) w[S[i]] = (1.0 - theta) * w[S[i]] + theta * y[i];
  w[S[drop]] = 0.0;
  int kept = 0;
  for (int i = 0; i < s; ++i) {
    if (w[S[i]] > kInside) S[kept++] = S[i];
    else w[S[i]] = 0.0;
  }
  return kept;
}

// ---------------------------------------------------------------------------
// MGDA
// ---------------------------------------------------------------------------

__device__ double pair_gamma(double gii, double gjj, double gij) {
  const double den = gii + gjj - 2.0 * gij;
  if (!(den > 0.0)) return 0.5;
  return fmin(1.0, fmax(0.0, (gjj - gij) / den));
}

// Best pair: the K=2 closed form on every pair, least value wins, ties to the
// first pair in lexicographic order.
__device__ void mgda_pair_start(int K, const double* G, double* al) {
  double best = 1e300, bg = 0.5;
  int bi = 0, bj = 1;
  for (int i = 0; i < K; ++i)
    for (int j = i + 1; j < K; ++j) {
      const double gii = G[i * K + i], gjj = G[j * K + j], gij = G[i * K + j];
      const double g = pair_gamma(gii, gjj, gij);
      const double val = g * g * gii + 2.0 * g * (1.0 - g) * gij + (1.0 - g) * (1.0 - g) * gjj;
      if (val < best) {
        best = val;
        bi = i;
        bj = j;
        bg = g;
      }
    }
  for (int k = 0; k < K; ++k) al[k] = 0.0;
  al[bi] = bg;
  al[bj] = 1.0 - bg;
}

// Frank-Wolfe with exact line search.  *met: stopped on the gap test.
__device__ void mgda_frank_wolfe(int K, const double* G, int max_iter, double tol, double* al,
                                 bool* met) {
  double v[kMaxK];
  *met = false;
  for (int it = 0; it < max_iter; ++it) {
    mat_vec(K, G, al, v);
    const double a = dotk(K, al, v);
    const int t = argmin_first(K, v);
    const double gap = a - v[t];
    if (gap <= tol) {
      *met = true;
      return;
    }
    const double den = a - 2.0 * v[t] + G[t * K + t];
    if (!(den > 0.0)) {
      *met = true;
      return;
    }
    const double g = fmin(1.0, gap / den);
    for (int k = 0; k < K; ++k) al[k] *= (1.0 - g);
    al[t] += g;
  }
}

// Exact completion from the support of al (Wolfe's corral iteration).
__device__ bool mgda_complete(int K, const double* G, double* al) {
  int S[kMaxK], s = 0;
  for (int k = 0; k < K; ++k) {
    if (al[k] > kInside) S[s++] = k;
    else al[k] = 0.0;
  }
  if (s == 0) return false;
  double y[kMaxK], v[kMaxK];
  for (int round = 0; round < 8 * K + 8; ++round) {
    if (!affine_min_norm(K, G, S, s, y)) return false;
    bool inside = true;
    for (int i = 0; i < s; ++i)
      if (!(y[i] > kInside)) inside = false;
    if (!inside) {
      s = step_to_boundary(al, S, s, y);
      if (s == 0) return false;
      continue;
    }
    for (int i = 0; i < s; ++i) al[S[i]] = y[i];
    mat_vec(K, G, al, v);
    const double xx = dotk(K, al, v);
    const int j = argmin_first(K, v);
    if (v[j] >= xx - kKkt) return true;
    for (int i = 0; i < s; ++i)
      if (S[i] == j) return true;
    S[s++] = j;
    al[j] = 0.0;
  }
  return false;
}

__device__ int solve_mgda(int K, const double* G, const SolveParams& p, double* beta) {
  if (K == 1) {
    beta[0] = 1.0;
    return BKMOO_OK;
  }
  if (K == 2 && (p.flags & BKMOO_FLAG_CLOSED_FORM_K2)) {
    const double g = pair_gamma(G[0], G[3], G[1]);
    beta[0] = g;
    beta[1] = 1.0 - g;
    return BKMOO_OK;
  }
  double al[kMaxK], keep[kMaxK];
  mgda_pair_start(K, G, al);
  bool met;
  mgda_frank_wolfe(K, G, p.max_iter, p.tol, al, &met);
  if (p.flags & BKMOO_FLAG_POLISH) {
    for (int k = 0; k < K; ++k) keep[k] = al[k];
    if (mgda_complete(K, G, al)) {
      double s = 0.0;
      for (int k = 0; k < K; ++k) s += al[k];
      for (int k = 0; k < K; ++k) beta[k] = al[k] / s;
      return BKMOO_OK;
    }
    for (int k = 0; k < K; ++k) al[k] = keep[k];
  }
  for (int k = 0; k < K; ++k) beta[k] = al[k];
  return met ? BKMOO_OK : BKMOO_ERR_NOT_CONVERGED;
}

// ---------------------------------------------------------------------------
// PCGrad
// ---------------------------------------------------------------------------

// SplitMix64 output function (Steele, Lea, Flood, OOPSLA 2014).
__device__ __forceinline__ uint64_t splitmix_out(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

__device__ void task_order(uint64_t seed, uint64_t step, int64_t b, int K, int t, int* order) {
  constexpr uint64_t kGamma = 0x9E3779B97F4A7C15ull;
  uint64_t key = splitmix_out(seed + (step + 1) * kGamma);
  key = splitmix_out(key + ((uint64_t)b + 1) * kGamma);
  key = splitmix_out(key + ((uint64_t)t + 1) * kGamma);
  int m = 0;
  for (int k = 0; k < K; ++k)
    if (k != t) order[m++] = k;
  uint64_t n = 1;
  for (int i = m - 1; i >= 1; --i, ++n) {
    const uint64_t r = splitmix_out(key + n * kGamma);
    const int j = (int)(r % (uint64_t)(i + 1));
    const int tmp = order[i];
    order[i] = order[j];
    order[j] = tmp;
  }
}

__device__ int solve_pcgrad(int K, const double* G, const SolveParams& p, int64_t b,
                            double* beta) {
  double row[kMaxK];
  int order[kMaxK];
  for (int k = 0; k < K; ++k) beta[k] = 0.0;
  for (int t = 0; t < K; ++t) {
    for (int k = 0; k < K; ++k) row[k] = (k == t) ? 1.0 : 0.0;
    task_order(p.seed, p.step, b, K, t, order);
    for (int q = 0; q < K - 1; ++q) {
      const int j = order[q];
      double pr = 0.0;
      for (int m = 0; m < K; ++m) pr += row[m] * G[m * K + j];
      const double gjj = G[j * K + j];
      if (pr < 0.0 && gjj > 0.0) row[j] -= pr / gjj;
    }
    for (int k = 0; k < K; ++k) beta[k] += row[k];
  }
  return BKMOO_OK;
}

// ---------------------------------------------------------------------------
// CAGrad
// ---------------------------------------------------------------------------

struct Cag {
  int K;
  const double* G;
  double b[kMaxK];  // b_k = <g_k, g0>
  double rho;       // c ||g0||
};

__device__ double cag_value(const Cag& c, const double* w) {
  double v[kMaxK];
  mat_vec(c.K, c.G, w, v);
  const double q = dotk(c.K, w, v);
  return dotk(c.K, c.b, w) + c.rho * sqrt(fmax(q, 0.0));
}

// Exact minimiser over [0, 1] of phi(g) = g L + rho sqrt(q + 2 A1 g + A2 g^2)
// (convex): the interior stationary point, the kink where the segment passes
// closest to the origin, and the two ends are compared.
__device__ double cag_line(double L, double q, double A1, double A2, double rho) {
  auto phi = [&](double g) {
    const double qq = q + 2.0 * A1 * g + A2 * g * g;
    return g * L + rho * sqrt(fmax(qq, 0.0));
  };
  double bestg = 0.0, best = phi(0.0);
  const double f1 = phi(1.0);
  if (f1 < best) {
    best = f1;
    bestg = 1.0;
  }
  if (A2 > 0.0) {
    const double D = fmax(A2 * q - A1 * A1, 0.0);
    const double kap = -L / (rho * sqrt(A2));
    if (fabs(kap) < 1.0) {
      const double u = kap * sqrt(D / (1.0 - kap * kap));
      const double g = (u - A1) / A2;
      if (g > 0.0 && g < 1.0) {
        const double f = phi(g);
        if (f < best) {
          best = f;
          bestg = g;
        }
      }
    }
    const double g0 = -A1 / A2;
    if (g0 > 0.0 && g0 < 1.0) {
      const double f = phi(g0);
      if (f < best) {
        best = f;
        bestg = g0;
      }
    }
  }
  return bestg;
}

// Stationary point of F on the affine hull of S: with m = G_SS^-1 1,
// n = G_SS^-1 b_S, D = (1^T n)^2 - (1^T m)(n^T b_S - rho^2) and
// lambda = (1^T n + sqrt D) / 1^T m, z = (lambda m - n) / sqrt D.
__device__ bool cag_affine(const Cag& c, const int* S, int s, double* z) {
  if (s == 1) {
    z[0] = 1.0;
    return true;
  }
  const int K = c.K, n = s + 2;
  double A[kMaxK * (kMaxK + 2)];
  for (int i = 0; i < s; ++i) {
    for (int j = 0; j < s; ++j) A[i * n + j] = c.G[S[i] * K + S[j]];
    A[i * n + s] = 1.0;
    A[i * n + s + 1] = c.b[S[i]];
  }
  if (!gauss_jordan(A, s, 2)) return false;
  double om = 0.0, on = 0.0, nb = 0.0;
  for (int i = 0; i < s; ++i) {
    om += A[i * n + s];
    on += A[i * n + s + 1];
    nb += A[i * n + s + 1] * c.b[S[i]];
  }
  const double D = on * on - om * (nb - c.rho * c.rho);
  if (!(om > 0.0) || !(D > 0.0)) return false;
  const double sd = sqrt(D);
  const double lam = (on + sd) / om;
  for (int i = 0; i < s; ++i) z[i] = (lam * A[i * n + s] - A[i * n + s + 1]) / sd;
  return true;
}

__device__ bool cag_complete(const Cag& c, double* w) {
  const int K = c.K;
  int S[kMaxK], s = 0;
  for (int k = 0; k < K; ++k) {
    if (w[k] > kInside) S[s++] = k;
    else w[k] = 0.0;
  }
  if (s == 0) return false;
  double z[kMaxK], v[kMaxK];
  for (int round = 0; round < 8 * K + 8; ++round) {
    if (!cag_affine(c, S, s, z)) return false;
    bool inside = true;
    for (int i = 0; i < s; ++i)
      if (!(z[i] > kInside)) inside = false;
    if (!inside) {
      s = step_to_boundary(w, S, s, z);
      if (s == 0) return false;
      continue;
    }
    double sum = 0.0;
    for (int i = 0; i < s; ++i) sum += z[i];
    for (int i = 0; i < s; ++i) w[S[i]] = z[i] / sum;
    mat_vec(K, c.G, w, v);
    const double q = dotk(K, w, v);
    if (!(q > 1e-24)) return false;
    const double nq = sqrt(q);
    double grad[kMaxK];
    for (int k = 0; k < K; ++k) grad[k] = c.b[k] + c.rho * v[k] / nq;
    const double lam = dotk(K, w, grad);
    const int j = argmin_first(K, grad);
    if (grad[j] >= lam - kKkt) return true;
    for (int i = 0; i < s; ++i)
      if (S[i] == j) return true;
    S[s++] = j;
    w[j] = 0.0;
  }
  return false;
}

__device__ int solve_cagrad(int K, const double* G, const SolveParams& p, double* beta) {
  Cag c;
  c.K = K;
  c.G = G;
  double tot = 0.0;
  for (int i = 0; i < K; ++i) {
    double r = 0.0;
    for (int j = 0; j < K; ++j) r += G[i * K + j];
    c.b[i] = r / K;
    tot += r;
  }
  const double g0sq = tot / ((double)K * K);
  for (int k = 0; k < K; ++k) beta[k] = 1.0 / K;
  if (!(p.cagrad_c > 0.0) || !(g0sq > 0.0)) return BKMOO_OK;
  c.rho = p.cagrad_c * sqrt(g0sq);

  double w[kMaxK], v[kMaxK], keep[kMaxK];
  int k0 = 0;
  double f0 = 1e300;
  for (int k = 0; k < K; ++k) {
    const double f = c.b[k] + c.rho * sqrt(fmax(G[k * K + k], 0.0));
    if (f < f0) {
      f0 = f;
      k0 = k;
    }
  }
  for (int k = 0; k < K; ++k) w[k] = (k == k0) ? 1.0 : 0.0;

  bool met = false;
  for (int it = 0; it < p.max_iter; ++it) {
    mat_vec(K, G, w, v);
    const double q = dotk(K, w, v);
    const double nq = sqrt(fmax(q, 0.0));
    if (!(nq > 1e-12)) {
      met = true;
      break;
    }
    const double bw = dotk(K, c.b, w);
    int t = 0;
    double gt = 1e300;
    for (int k = 0; k < K; ++k) {
      const double gk = c.b[k] + c.rho * v[k] / nq;
      if (gk < gt) {
        gt = gk;
        t = k;
      }
    }
    const double gap = bw + c.rho * nq - gt;
    if (gap <= p.tol) {
      met = true;
      break;
    }
    const double L = c.b[t] - bw, A1 = v[t] - q, A2 = q - 2.0 * v[t] + G[t * K + t];
    const double g = cag_line(L, q, A1, A2, c.rho);
    if (!(g > 0.0)) {
      met = true;
      break;
    }
    for (int k = 0; k < K; ++k) w[k] *= (1.0 - g);
    w[t] += g;
  }
  if (p.flags & BKMOO_FLAG_POLISH) {
    for (int k = 0; k < K; ++k) keep[k] = w[k];
    const double fk = cag_value(c, w);
    if (cag_complete(c, w) && cag_value(c, w) <= fk + 1e-15 * fabs(fk) + 1e-300) {
      met = true;
    } else {
      for (int k = 0; k < K; ++k) w[k] = keep[k];
    }
  }
  mat_vec(K, G, w, v);
  const double q = dotk(K, w, v);
  if (q > 1e-24) {
    const double f = c.rho / sqrt(q);
    for (int k = 0; k < K; ++k) beta[k] = 1.0 / K + f * w[k];
  }
  return met ? BKMOO_OK : BKMOO_ERR_NOT_CONVERGED;
}

// ---------------------------------------------------------------------------
// per bucket
// ---------------------------------------------------------------------------

__device__ int solve_bucket(int K, double* G, const SolveParams& p, int64_t b, double* beta) {
  bool finite = true;
  double scale = 0.0;
  for (int i = 0; i < K * K; ++i)
    if (!isfinite(G[i])) finite = false;
  if (!finite) {
    for (int k = 0; k < K; ++k) beta[k] = 1.0 / K;
    return BKMOO_ERR_NONFINITE;
  }
  for (int k = 0; k < K; ++k) scale = fmax(scale, G[k * K + k]);
  if (scale > 0.0) {
    const double inv = 1.0 / scale;
    for (int i = 0; i < K * K; ++i) G[i] *= inv;
  }
  switch (p.rule) {
    case BKMOO_MGDA:
      return solve_mgda(K, G, p, beta);
    case BKMOO_PCGRAD:
      return solve_pcgrad(K, G, p, b, beta);
    case BKMOO_CAGRAD:
      return solve_cagrad(K, G, p, beta);
    default:
      for (int k = 0; k < K; ++k) beta[k] = 1.0 / K;
      return BKMOO_OK;
  }
}

__global__ void __launch_bounds__(32 * kSolveWarpsPerBlock)
    solve_kernel(const PlanView v, const SolveParams p, float* out_weights,
                 int32_t* out_status) {
  __shared__ double Gs[kSolveWarpsPerBlock][kMaxK * kMaxK];
  const int lane = threadIdx.x & 31, wi = threadIdx.x >> 5;
  const int64_t b = (int64_t)blockIdx.x * kSolveWarpsPerBlock + wi;
  if (b >= v.n_buckets) return;
  const int K = v.K;
  if (!header_ok(v)) {
    if (lane == 0 && out_status) out_status[b] = BKMOO_ERR_WORKSPACE;
    return;
  }
  double* G = Gs[wi];
  reduce_bucket(v, b, G, lane);
  if (lane != 0) return;
  double beta[kMaxK];
  const int st = solve_bucket(K, G, p, b, beta);
  for (int k = 0; k < K; ++k) {
    const float f = (float)beta[k];
    v.beta[b * K + k] = f;
    if (out_weights) out_weights[b * K + k] = f;
  }
  if (out_status) out_status[b] = st;
}

__global__ void __launch_bounds__(32 * kSolveWarpsPerBlock)
    gram_finalize_kernel(const PlanView v, double* out_gram) {
  __shared__ double Gs[kSolveWarpsPerBlock][kMaxK * kMaxK];
  const int lane = threadIdx.x & 31, wi = threadIdx.x >> 5;
  const int64_t b = (int64_t)blockIdx.x * kSolveWarpsPerBlock + wi;
  if (b >= v.n_buckets) return;
  if (!header_ok(v)) return;
  const int K = v.K;
  double* G = Gs[wi];
  reduce_bucket(v, b, G, lane);
  for (int i = lane; i < K * K; i += 32) out_gram[b * K * K + i] = G[i];
}

}  // namespace

cudaError_t launch_solve(const PlanView& v, const SolveParams& p, float* out_weights,
                         int32_t* out_status, cudaStream_t s) {
  if (v.n_buckets == 0) return cudaSuccess;
  const int64_t grid = (v.n_buckets + kSolveWarpsPerBlock - 1) / kSolveWarpsPerBlock;
  solve_kernel<<<(unsigned)grid, 32 * kSolveWarpsPerBlock, 0, s>>>(v, p, out_weights, out_status);
  return cudaGetLastError();
}

cudaError_t launch_gram_finalize(const PlanView& v, double* out_gram, cudaStream_t s) {
  if (v.n_buckets == 0) return cudaSuccess;
  const int64_t grid = (v.n_buckets + kSolveWarpsPerBlock - 1) / kSolveWarpsPerBlock;
  gram_finalize_kernel<<<(unsigned)grid, 32 * kSolveWarpsPerBlock, 0, s>>>(v, out_gram);
  return cudaGetLastError();
}

}  // namespace bkmoo
