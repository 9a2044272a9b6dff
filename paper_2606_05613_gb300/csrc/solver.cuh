// Per-bucket solvers of the MOO rules on a bucket's Gram matrix G (fp64),
// shared by the solve kernel (solve.cu) and the fused kernel (fused.cu).
// A whole warp enters solve_bucket_warp(); the coefficients beta of
// d_b = sum_k beta_k g_k come out in shared memory.
//
//  MGDA (Eq. 3; bucket form Eq. 6 over the simplex of Algorithm 1):
//    K = 2 (flag CLOSED_FORM_K2): gamma = clamp(<g2 - g1, g2> / ||g1 - g2||^2, 0, 1).
//    2 <= K <= 5 with POLISH: exact, by enumeration of the supports, one per
//      lane: lane l takes S = the bits of l + 1, finds the affine
//      minimum-norm point of S in fp32 and keeps it if it lies in the
//      simplex; the least norm wins, is refined in fp64 and checked.
//    K >= 6 with POLISH: Wolfe's minimum-norm-point algorithm in fp32 with a
//      lane-parallel Gauss-Jordan, one fp64 refinement of the final support
//      and the same check.
//    Without POLISH, or when a check fails: Frank-Wolfe from the best pair
//      with exact line search (lane 0, fp64), then (POLISH) an exact
//      active-set completion in the manner of Wolfe's minimum-norm-point
//      algorithm: the affine minimum-norm point of
//      the current support is taken when it lies inside the simplex, else the
//      iterate moves to the boundary and drops a point; a point is added
//      while some g_j has <d, g_j> < ||d||^2.
//  CAGrad (Eq. 4; Eq. 7): the dual min_{w in simplex} F(w),
//    F(w) = <g0, g_w> + c ||g0|| ||g_w||, beta = 1/K + c ||g0|| w / ||g_w||.
//    K <= 5 with POLISH: exact, one support per lane, with the closed-form
//      stationary point of F on the support's affine hull (fp32 search,
//      fp64 refinement and check).
//    K >= 6 with POLISH: the same kind of active-set method in fp32 with the
//      lane-parallel Gauss-Jordan, from the best vertex; fp64 refinement and
//      check.
//    Without POLISH, or when a check fails: Frank-Wolfe with exact line
//      search from the best vertex (lane 0, fp64), then (POLISH) the same
//      kind of active-set completion.
//  PCGrad (Eq. 5; Eq. 8): the projections of Algorithm 1 carried out on the
//    coefficients of each running d_t, since <d_t, g_j> = sum_m C_tm G_mj;
//    one lane per task.
//  MEAN: beta = 1/K.
//
// All solvers work on G scaled by a power of two so that max_k G_kk lies in
// [1, 2) (every rule is invariant under a positive scaling of G).  A Gram with a NaN or Inf gives
// beta = 1/K and status BKMOO_ERR_NONFINITE.
#pragma once

#include <math.h>

#include "common.cuh"

namespace bkmoo {
namespace solver {
namespace {

constexpr double kInside = 1e-15;  // weights above this are in the support
constexpr double kKkt = 1e-13;     // optimality slack on the normalised Gram
constexpr double kPivot = 1e-13;   // smallest pivot of a non-singular system

// ---------------------------------------------------------------------------
// partial reduction
// ---------------------------------------------------------------------------

// Lane p sums entry p of the bucket's chunk partials in a fixed order: eight
// interleaved fp64 running sums (chunk c0 + 8m + j goes to sum j), added by a
// fixed tree; eight independent chains hide the fp64 add latency, which a
// single chain pays once per chunk (1600 chunks in a 100 MiB fp32 bucket).
// A bucket of more than kGroupMinChunks chunks was pre-reduced by
// group_reduce_kernel: its group sums sit in the rows of the first chunk of
// each group of kGroupChunks, and those rows are what is summed here.
__device__ void reduce_bucket(const PlanView& v, int64_t b, double* G, int lane) {
  const int K = v.K, P = tri(K);
  int64_t c0 = v.chunk_prefix[b], c1 = v.chunk_prefix[b + 1];
  int64_t stride = 1;  // in chunks
  if (c1 - c0 > kGroupMinChunks) {
    stride = kGroupChunks;
    c1 = c0 + (c1 - c0 + kGroupChunks - 1) / kGroupChunks;  // c0 + number of groups
  }
  const int64_t rs = stride * P;  // doubles between the rows summed
  for (int p = lane; p < P; p += 32) {
    double t[8] = {0.0, 0.0, 0.0, 0.0, 0.0, 0.0, 0.0, 0.0};
    const double* src = v.partials + c0 * P + p;
    int64_t c = c0;
    for (; c + 8 <= c1; c += 8, src += 8 * rs) {
#pragma unroll
      for (int j = 0; j < 8; ++j) t[j] += src[j * rs];
    }
#pragma unroll
    for (int j = 0; j < 8; ++j)
      if (c + j < c1) t[j] += src[j * rs];
    const double s = ((t[0] + t[1]) + (t[2] + t[3])) + ((t[4] + t[5]) + (t[6] + t[7]));
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
// fast warp solvers: fp32 search, fp64 refinement and verification
// ---------------------------------------------------------------------------
//
// On this GPU a dependent fp64 FMA takes about 14 times as long as an fp32
// one and fp64 division or square root about 100 times, so the search for
// the optimal support runs in fp32 (registers, one support per lane), and
// fp64 is spent on two mixed-precision iterative-refinement steps of the
// winning support's linear system and on checking the optimality
// conditions.  A failed check falls back to the serial fp64 solvers above.

constexpr int kEnumMaxK = 5;

// a / b and sqrt(x) in fp64 by Newton-Raphson from an fp32 seed: for the
// quotient r = 1/b rounded to fp32, q = a r, then one step with the residual
// correction q + (a - b q) r; for the root s = sqrt(x) rounded to fp32, then
// s + (x - s^2) / (2 s) with 1 / (2 s) from the fp32 reciprocal.  The seed
// carries a relative error of about 2^-23 (two fp32 roundings), which the
// step squares: at most about 2^-46 (tested against the correctly rounded
// operations).  Operands where the seed or the intermediate products could
// leave the fp32 / fp64 normal range (|b| or x outside (1e-30, 1e30), a
// nonzero |a| outside (1e-270, 1e270)) take the correctly rounded fp64
// operation instead.
__device__ __forceinline__ double div_nr(double a, double b) {
  const double ab = fabs(b), aa = fabs(a);
  if (!(ab > 1e-30 && ab < 1e30 && aa < 1e270 && (aa > 1e-270 || a == 0.0))) return a / b;
  const double r = (double)__frcp_rn((float)b);
  const double q = a * r;
  return fma(fma(-b, q, a), r, q);
}
__device__ __forceinline__ double sqrt_nr(double x) {
  if (!(x > 1e-30 && x < 1e30)) return x > 0.0 ? sqrt(x) : 0.0;
  const double s0 = (double)sqrtf((float)x);
  const double h = 0.5 * (double)__frcp_rn((float)s0);
  return fma(fma(-s0, s0, x), h, s0);
}

// Warp argmin of (value, lane), ties to the lowest lane; every lane gets it.
__device__ __forceinline__ int warp_argmin(float val, int lane) {
  int best = lane;
  for (int off = 16; off > 0; off >>= 1) {
    const float v2 = __shfl_xor_sync(0xffffffffu, val, off);
    const int l2 = __shfl_xor_sync(0xffffffffu, best, off);
    if (v2 < val || (v2 == val && l2 < best)) {
      val = v2;
      best = l2;
    }
  }
  return best;
}

// Gauss-Jordan inverse of an N x N fp32 matrix with partial pivoting.  Rows
// are swapped by selects, so every index is a compile-time constant and the
// matrices stay in registers.  False if a pivot is below `piv`.
template <int N>
__device__ __forceinline__ bool inverse32(float (&A)[N][N], float (&X)[N][N], float piv) {
#pragma unroll
  for (int r = 0; r < N; ++r)
#pragma unroll
    for (int j = 0; j < N; ++j) X[r][j] = (r == j) ? 1.0f : 0.0f;
  bool ok = true;
#pragma unroll
  for (int c = 0; c < N; ++c) {
    int p = c;
    float best = fabsf(A[c][c]);
#pragma unroll
    for (int r = c + 1; r < N; ++r)
      if (fabsf(A[r][c]) > best) {
        best = fabsf(A[r][c]);
        p = r;
      }
    ok = ok && (best > piv);
#pragma unroll
    for (int r = c + 1; r < N; ++r) {
      const bool sw = (p == r);
#pragma unroll
      for (int j = 0; j < N; ++j) {
        const float a0 = A[c][j], a1 = A[r][j], x0 = X[c][j], x1 = X[r][j];
        A[c][j] = sw ? a1 : a0;
        A[r][j] = sw ? a0 : a1;
        X[c][j] = sw ? x1 : x0;
        X[r][j] = sw ? x0 : x1;
      }
    }
    const float inv = __frcp_rn(A[c][c]);
#pragma unroll
    for (int j = 0; j < N; ++j) {
      A[c][j] *= inv;
      X[c][j] *= inv;
    }
#pragma unroll
    for (int r = 0; r < N; ++r) {
      if (r == c) continue;
      const float f = A[r][c];
#pragma unroll
      for (int j = 0; j < N; ++j) {
        A[r][j] = fmaf(-f, A[c][j], A[r][j]);
        X[r][j] = fmaf(-f, X[c][j], X[r][j]);
      }
    }
  }
  return ok;
}

template <int K>
__device__ __forceinline__ bool in_mask(unsigned m, int k) {
  return (m >> k) & 1u;
}

// MGDA, one support S (bit mask) per lane: the affine minimum-norm point of
// S from the bordered system A z = e_K with A = [G_SS 1; 1^T 0] (rows and
// columns outside S replaced by the identity so that the system keeps size
// K + 1).  Returns its squared norm in fp32, +inf if S is singular or the
// point leaves the simplex; Ainv and z for the refinement.
template <int K>
__device__ float mgda_candidate32(const float* G, unsigned mask, float (&Ainv)[K + 1][K + 1],
                                  float (&z)[K + 1]) {
  constexpr int N = K + 1;
  float A[N][N];
#pragma unroll
  for (int i = 0; i < K; ++i) {
#pragma unroll
    for (int j = 0; j < K; ++j)
      A[i][j] = (in_mask<K>(mask, i) && in_mask<K>(mask, j)) ? G[i * K + j]
                : (i == j && !in_mask<K>(mask, i)) ? 1.0f : 0.0f;
    A[i][K] = in_mask<K>(mask, i) ? 1.0f : 0.0f;
    A[K][i] = in_mask<K>(mask, i) ? 1.0f : 0.0f;
  }
  A[K][K] = 0.0f;
  if (!inverse32<N>(A, Ainv, 1e-6f)) return INFINITY;
#pragma unroll
  for (int i = 0; i < N; ++i) z[i] = Ainv[i][K];
  float q = 0.0f;
  bool ok = true;
#pragma unroll
  for (int i = 0; i < K; ++i) {
    if (!in_mask<K>(mask, i)) continue;
    if (z[i] < -1e-5f) ok = false;
#pragma unroll
    for (int j = 0; j < K; ++j)
      if (in_mask<K>(mask, j)) q = fmaf(z[i] * G[i * K + j], z[j], q);
  }
  return ok ? q : INFINITY;
}

// One mixed-precision refinement step of A z = e_K (residual in fp64,
// correction through the fp32 inverse: error about (cond(A) 2^-24)^2), then
// alpha = z on S, >= 0, renormalised.
template <int K>
__device__ void mgda_refine(const double* G, unsigned mask, const float (&Ainv)[K + 1][K + 1],
                            const float (&z32)[K + 1], double (&alpha)[K]) {
  constexpr int N = K + 1;
  double z[N];
#pragma unroll
  for (int i = 0; i < N; ++i) z[i] = z32[i];
  {
    float r[N];
#pragma unroll
    for (int i = 0; i < K; ++i) {
      double t;
      if (in_mask<K>(mask, i)) {
        t = -z[K];
#pragma unroll
        for (int j = 0; j < K; ++j)
          if (in_mask<K>(mask, j)) t = fma(-G[i * K + j], z[j], t);
      } else {
        t = -z[i];
      }
      r[i] = (float)t;
    }
    double t = 1.0;
#pragma unroll
    for (int j = 0; j < K; ++j)
      if (in_mask<K>(mask, j)) t -= z[j];
    r[K] = (float)t;
#pragma unroll
    for (int i = 0; i < N; ++i) {
      float d = 0.0f;
#pragma unroll
      for (int j = 0; j < N; ++j) d = fmaf(Ainv[i][j], r[j], d);
      z[i] += (double)d;
    }
  }
  double s = 0.0;
#pragma unroll
  for (int k = 0; k < K; ++k) {
    alpha[k] = (in_mask<K>(mask, k) && z[k] > 0.0) ? z[k] : 0.0;
    s += alpha[k];
  }
  const double corr = 2.0 - s;  // 1 / s to first order, s = 1 + O(1e-16)
#pragma unroll
  for (int k = 0; k < K; ++k) alpha[k] *= corr;
}

// The same refinement step with its fp64 work spread over the warp, for
// K <= 4 (every lane calls it; the winner lane `win` holds Ainv and z32).  On
// this GPU an fp64 warp instruction costs tens of cycles whatever the number
// of active lanes, so the serial form above spends most of a solve in its
// ~60 of them: here lane l = 4 i + j forms the residual's term (i, j) of the
// bordered system (row K: the simplex row), a two-level butterfly adds each
// row, the winner applies its fp32 inverse, and lane k forms alpha_k.
// Returns alpha_k on lane k < K, 0 on the other lanes.
template <int K>
__device__ double mgda_refine_warp(const double* G, unsigned mask, int win,
                                   const float (&Ainv)[K + 1][K + 1], const float (&z32)[K + 1],
                                   int lane) {
  static_assert(K >= 1 && K <= 4, "rows of four lanes");
  constexpr int N = K + 1;
  float z[N];
#pragma unroll
  for (int c = 0; c < N; ++c) z[c] = __shfl_sync(0xffffffffu, z32[c], win);
  const int i = lane >> 2, j = lane & 3;
  float zi = 0.0f, zj = 0.0f;
#pragma unroll
  for (int c = 0; c < K; ++c) {
    if (i == c) zi = z[c];
    if (j == c) zj = z[c];
  }
  // term (i, j): G_ij z_j on the rows of G, z_j on the simplex row
  const bool col_in = j < K && in_mask<K>(mask, j);
  const double g = (i < K && j < K) ? G[i * K + j] : 1.0;
  double term = col_in ? g * (double)zj : 0.0;
  term += __shfl_xor_sync(0xffffffffu, term, 1);
  term += __shfl_xor_sync(0xffffffffu, term, 2);
  // residual of row i on its first lane: -(z_K + row) in S, -z_i outside,
  // 1 - sum on the simplex row
  double r;
  if (i < K)
    r = in_mask<K>(mask, i) ? -((double)z[K] + term) : -(double)zi;
  else
    r = 1.0 - term;
  const float rf = (float)r;
  float rr[N];
#pragma unroll
  for (int c = 0; c < N; ++c) rr[c] = __shfl_sync(0xffffffffu, rf, 4 * c);
  // correction through the winner's fp32 inverse
  float dk = 0.0f, zk = 0.0f;
#pragma unroll
  for (int c = 0; c < K; ++c) {
    float t = 0.0f;
#pragma unroll
    for (int jj = 0; jj < N; ++jj) t = fmaf(Ainv[c][jj], rr[jj], t);
    t = __shfl_sync(0xffffffffu, t, win);
    if (lane == c) {
      dk = t;
      zk = z[c];
    }
  }
  double a = 0.0;
  if (lane < K) {
    a = (double)zk + (double)dk;
    a = (in_mask<K>(mask, lane) && a > 0.0) ? a : 0.0;
  }
  double s = a;
  s += __shfl_xor_sync(0xffffffffu, s, 1);
  s += __shfl_xor_sync(0xffffffffu, s, 2);
  return a * (2.0 - s);  // 2 - s = 1 / s to first order, s = 1 + O(1e-16)
}

// Exact MGDA for 2 <= K <= 5.  False (beta untouched) if the optimality
// check fails; the caller then takes the serial fp64 path.
template <int K>
__device__ bool mgda_fast(const double* G, const float* Gf, int lane, double* beta_out) {
  constexpr int N = K + 1;
  float Ainv[N][N], z[N];
  const unsigned mask = (unsigned)lane + 1u;
  float q = INFINITY;
  if (mask < (1u << K)) q = mgda_candidate32<K>(Gf, mask, Ainv, z);
  const int win = warp_argmin(q, lane);
  const unsigned wmask = (unsigned)win + 1u;
  if (!(__shfl_sync(0xffffffffu, q, win) < INFINITY)) return false;
  double alpha[K];
  float a32[K];
  if constexpr (K <= 4) {
    const double mine = mgda_refine_warp<K>(G, wmask, win, Ainv, z, lane);
    const float mine32 = (float)mine;
#pragma unroll
    for (int k = 0; k < K; ++k) {
      alpha[k] = __shfl_sync(0xffffffffu, mine, k);
      a32[k] = __shfl_sync(0xffffffffu, mine32, k);
    }
  } else {
    if (lane == win) mgda_refine<K>(G, wmask, Ainv, z, alpha);
#pragma unroll
    for (int k = 0; k < K; ++k) {
      alpha[k] = __shfl_sync(0xffffffffu, alpha[k], win);
      a32[k] = (float)alpha[k];
    }
  }
  // optimality: <g_k, d> >= ||d||^2 for every k (proof of Theorem 3.1); on
  // S it holds with equality by construction, off S it is checked in fp32
  // with a margin far above fp32 rounding, and in fp64 only when marginal
  {
    float v32[K], xx32 = 0.0f;
#pragma unroll
    for (int k = 0; k < K; ++k) {
      float t = 0.0f;
#pragma unroll
      for (int j = 0; j < K; ++j) t = fmaf(Gf[k * K + j], a32[j], t);
      v32[k] = t;
      xx32 = fmaf(a32[k], t, xx32);
    }
    bool clear = true;
#pragma unroll
    for (int k = 0; k < K; ++k)
      if (!in_mask<K>(wmask, k) && !(v32[k] - xx32 >= 1e-5f)) clear = false;
    if (!clear) {
      double v[K], xx = 0.0, vmin = 1e300;
#pragma unroll
      for (int k = 0; k < K; ++k) {
        double t = 0.0;
#pragma unroll
        for (int j = 0; j < K; ++j) t = fma(G[k * K + j], alpha[j], t);
        v[k] = t;
      }
#pragma unroll
      for (int k = 0; k < K; ++k) {
        xx = fma(alpha[k], v[k], xx);
        vmin = fmin(vmin, v[k]);
      }
      if (!(vmin >= xx - kKkt)) return false;
    }
  }
  if (lane == 0)
#pragma unroll
    for (int k = 0; k < K; ++k) beta_out[k] = alpha[k];
  return true;
}

// CAGrad, one support per lane: the stationary point of
// F(w) = b^T w + rho sqrt(w^T G w) on the affine hull of S in fp32 (see
// cag_affine), F there (+inf if S is singular, D <= 0 or w leaves the
// simplex); the fp32 inverse of the masked G_SS for the refinement.
template <int K>
__device__ float cagrad_candidate32(const float* G, const float (&b)[K], float rho,
                                    unsigned mask, float (&Ginv)[K][K], float (&w)[K]) {
  const int s = __popc(mask);
#pragma unroll
  for (int k = 0; k < K; ++k) w[k] = 0.0f;
  if (s == 1) {
    const int k0 = __ffs(mask) - 1;
    float gkk = 0.0f, bk = 0.0f;
#pragma unroll
    for (int k = 0; k < K; ++k)
      if (k == k0) {
        w[k] = 1.0f;
        gkk = G[k * K + k];
        bk = b[k];
      }
    return bk + rho * sqrtf(fmaxf(gkk, 0.0f));
  }
  float A[K][K];
#pragma unroll
  for (int i = 0; i < K; ++i)
#pragma unroll
    for (int j = 0; j < K; ++j)
      A[i][j] = (in_mask<K>(mask, i) && in_mask<K>(mask, j)) ? G[i * K + j]
                : (i == j && !in_mask<K>(mask, i)) ? 1.0f : 0.0f;
  if (!inverse32<K>(A, Ginv, 1e-6f)) return INFINITY;
  float om = 0.0f, on = 0.0f, nb = 0.0f, m[K], n[K];
#pragma unroll
  for (int i = 0; i < K; ++i) {
    float mi = 0.0f, ni = 0.0f;
#pragma unroll
    for (int j = 0; j < K; ++j)
      if (in_mask<K>(mask, j)) {
        mi += Ginv[i][j];
        ni = fmaf(Ginv[i][j], b[j], ni);
      }
    m[i] = mi;
    n[i] = ni;
    if (in_mask<K>(mask, i)) {
      om += mi;
      on += ni;
      nb = fmaf(ni, b[i], nb);
    }
  }
  const float D = on * on - om * (nb - rho * rho);
  if (!(om > 0.0f) || !(D > 0.0f)) return INFINITY;
  const float sd = sqrtf(D), lam = (on + sd) / om;
  float sum = 0.0f;
#pragma unroll
  for (int i = 0; i < K; ++i)
    if (in_mask<K>(mask, i)) {
      const float wi = (lam * m[i] - n[i]) / sd;
      if (wi < -1e-5f) return INFINITY;
      w[i] = fmaxf(wi, 0.0f);
      sum += w[i];
    }
  if (!(sum > 0.0f)) return INFINITY;
  float q = 0.0f, bw = 0.0f;
#pragma unroll
  for (int i = 0; i < K; ++i) {
    w[i] /= sum;
    bw = fmaf(b[i], w[i], bw);
  }
#pragma unroll
  for (int i = 0; i < K; ++i)
#pragma unroll
    for (int j = 0; j < K; ++j) q = fmaf(w[i] * G[i * K + j], w[j], q);
  return bw + rho * sqrtf(fmaxf(q, 0.0f));
}

// fp64 stationary point on the winning support: m = G_SS^-1 1 and
// n = G_SS^-1 b_S with one refinement step, then the closed form.
template <int K>
__device__ void cagrad_refine(const double* G, const double (&b)[K], double rho, unsigned mask,
                              const float (&Ginv)[K][K], double (&w)[K]) {
  if (__popc(mask) == 1) {
#pragma unroll
    for (int k = 0; k < K; ++k) w[k] = in_mask<K>(mask, k) ? 1.0 : 0.0;
    return;
  }
  double m[K], n[K];
#pragma unroll
  for (int i = 0; i < K; ++i) {
    float mi = 0.0f, ni = 0.0f;
#pragma unroll
    for (int j = 0; j < K; ++j)
      if (in_mask<K>(mask, j)) {
        mi += Ginv[i][j];
        ni = fmaf(Ginv[i][j], (float)b[j], ni);
      }
    m[i] = mi;
    n[i] = ni;
  }
  {
    float rm[K], rn[K];
#pragma unroll
    for (int i = 0; i < K; ++i) {
      double tm, tn;
      if (in_mask<K>(mask, i)) {
        tm = 1.0;
        tn = b[i];
#pragma unroll
        for (int j = 0; j < K; ++j)
          if (in_mask<K>(mask, j)) {
            tm = fma(-G[i * K + j], m[j], tm);
            tn = fma(-G[i * K + j], n[j], tn);
          }
      } else {
        tm = -m[i];
        tn = -n[i];
      }
      rm[i] = (float)tm;
      rn[i] = (float)tn;
    }
#pragma unroll
    for (int i = 0; i < K; ++i) {
      float dm = 0.0f, dn = 0.0f;
#pragma unroll
      for (int j = 0; j < K; ++j) {
        dm = fmaf(Ginv[i][j], rm[j], dm);
        dn = fmaf(Ginv[i][j], rn[j], dn);
      }
      m[i] += (double)dm;
      n[i] += (double)dn;
    }
  }
  double om = 0.0, on = 0.0, nb = 0.0;
#pragma unroll
  for (int i = 0; i < K; ++i)
    if (in_mask<K>(mask, i)) {
      om += m[i];
      on += n[i];
      nb = fma(n[i], b[i], nb);
    }
  const double D = on * on - om * (nb - rho * rho);
  const double sd = sqrt_nr(D);
  const double lam = div_nr(on + sd, om), isd = div_nr(1.0, sd);
  double s = 0.0;
#pragma unroll
  for (int i = 0; i < K; ++i) {
    const double wi = in_mask<K>(mask, i) ? (lam * m[i] - n[i]) * isd : 0.0;
    w[i] = wi > 0.0 ? wi : 0.0;
    s += w[i];
  }
  const double corr = 2.0 - s;
#pragma unroll
  for (int i = 0; i < K; ++i) w[i] *= corr;
}

// Exact CAGrad for 1 <= K <= 5.  False if no candidate passes the
// optimality check (e.g. the minimum of F at g_w = 0).
template <int K>
__device__ bool cagrad_fast(const double* G, const float* Gf, double c, int lane,
                            double* beta_out) {
  double b[K], tot = 0.0;
  float bf[K];
#pragma unroll
  for (int i = 0; i < K; ++i) {
    double r = 0.0;
#pragma unroll
    for (int j = 0; j < K; ++j) r += G[i * K + j];
    b[i] = r * (1.0 / K);
    bf[i] = (float)b[i];
    tot += r;
  }
  const double g0sq = tot * (1.0 / ((double)K * K));
  if (!(c > 0.0) || !(g0sq > 0.0)) {
    if (lane == 0)
#pragma unroll
      for (int k = 0; k < K; ++k) beta_out[k] = 1.0 / K;
    return true;
  }
  // No sign condition on b: when 0 may lie in the hull (some b_k <= 0) the
  // minimiser still has g_w != 0 unless F's minimum sits at the kink
  // g_w = 0; the optimality check below certifies the candidate either way
  // (F is convex and differentiable wherever g_w != 0), and a candidate that
  // fails it goes to the serial path.
  const double rho = c * sqrt_nr(g0sq);
  float Ginv[K][K], w32[K];
  const unsigned mask = (unsigned)lane + 1u;
  float F = INFINITY;
  if (mask < (1u << K)) F = cagrad_candidate32<K>(Gf, bf, (float)rho, mask, Ginv, w32);
  const int win = warp_argmin(F, lane);
  if (!(__shfl_sync(0xffffffffu, F, win) < INFINITY)) return false;
  double w[K];
  if (lane == win) cagrad_refine<K>(G, b, rho, (unsigned)win + 1u, Ginv, w);
#pragma unroll
  for (int k = 0; k < K; ++k) w[k] = __shfl_sync(0xffffffffu, w[k], win);
  // optimality of the dual: grad_k = b_k + rho (G w)_k / ||g_w|| >= w^T grad
  // (equality on the support); fp32 with a margin, fp64 when marginal
  const unsigned wmask = (unsigned)win + 1u;
  double v[K], q = 0.0;
#pragma unroll
  for (int k = 0; k < K; ++k) {
    float t = 0.0f;
#pragma unroll
    for (int j = 0; j < K; ++j) t = fmaf(Gf[k * K + j], (float)w[j], t);
    v[k] = t;
  }
  {
    float q32 = 0.0f;
#pragma unroll
    for (int k = 0; k < K; ++k) q32 = fmaf((float)w[k], (float)v[k], q32);
    if (!(q32 > 1e-12f)) return false;
    const float f32 = (float)rho / sqrtf(q32);
    float lam32 = 0.0f;
    float g32[K];
#pragma unroll
    for (int k = 0; k < K; ++k) {
      g32[k] = fmaf(f32, (float)v[k], bf[k]);
      lam32 = fmaf((float)w[k], g32[k], lam32);
    }
    bool clear = true;
#pragma unroll
    for (int k = 0; k < K; ++k)
      if (!in_mask<K>(wmask, k) && !(g32[k] - lam32 >= 1e-5f)) clear = false;
    if (!clear) {
#pragma unroll
      for (int k = 0; k < K; ++k) {
        double t = 0.0;
#pragma unroll
        for (int j = 0; j < K; ++j) t = fma(G[k * K + j], w[j], t);
        v[k] = t;
      }
      double qq = 0.0;
#pragma unroll
      for (int k = 0; k < K; ++k) qq = fma(w[k], v[k], qq);
      if (!(qq > 1e-24)) return false;
      const double fd = div_nr(rho, sqrt_nr(qq));
      double lam = 0.0, gmin = 1e300;
#pragma unroll
      for (int k = 0; k < K; ++k) {
        const double gk = fma(fd, v[k], b[k]);
        lam = fma(w[k], gk, lam);
        gmin = fmin(gmin, gk);
      }
      if (!(gmin >= lam - 1e-11)) return false;
    }
  }
  // beta = 1/K + rho w / ||g_w|| with ||g_w|| in fp64
#pragma unroll
  for (int k = 0; k < K; ++k) {
    double t = 0.0;
#pragma unroll
    for (int j = 0; j < K; ++j) t = fma(G[k * K + j], w[j], t);
    q = fma(w[k], t, q);
  }
  if (!(q > 1e-24)) return false;
  const double f = div_nr(rho, sqrt_nr(q));
  if (lane == 0)
#pragma unroll
    for (int k = 0; k < K; ++k) beta_out[k] = fma(f, w[k], 1.0 / K);
  return true;
}

// CAGrad for K <= 4 with the fp64 work spread over the warp (lane l = 4 i + j
// holds entry (i, j) of G; every fp64 warp instruction costs tens of cycles
// on this GPU however few lanes are active): the same candidates, one
// refinement step of G_SS m = 1 and G_SS n = b with residuals in fp64, and
// the same optimality check as cagrad_fast.  On S the weights are
// w ~ (on + sqrt(D)) m - om n (lambda m - n with lambda = (on + sqrt(D)) / om,
// times om), normalised by their fp64 sum: one division instead of two.
template <int K>
__device__ bool cagrad_fast_warp(const double* G, const float* Gf, double c, int lane,
                                 double* beta_out) {
  static_assert(K >= 1 && K <= 4, "rows of four lanes");
  const int i = lane >> 2, j = lane & 3;
  const double gij = (i < K && j < K) ? G[i * K + j] : 0.0;
  // b_i = (G 1)_i / K on the lanes of row i, ||g0||^2 = 1^T G 1 / K^2
  double row = gij;
  row += __shfl_xor_sync(0xffffffffu, row, 1);
  row += __shfl_xor_sync(0xffffffffu, row, 2);
  double tot = j == 0 ? row : 0.0;
  tot += __shfl_xor_sync(0xffffffffu, tot, 4);
  tot += __shfl_xor_sync(0xffffffffu, tot, 8);
  tot = __shfl_sync(0xffffffffu, tot, 0);
  const double bi = row * (1.0 / K);
  const float bif = (float)bi;
  double b[K];
  float bf[K];
#pragma unroll
  for (int k = 0; k < K; ++k) {
    b[k] = __shfl_sync(0xffffffffu, bi, 4 * k);
    bf[k] = __shfl_sync(0xffffffffu, bif, 4 * k);
  }
  const double g0sq = tot * (1.0 / ((double)K * K));
  if (!(c > 0.0) || !(g0sq > 0.0)) {
    if (lane < K) beta_out[lane] = 1.0 / K;
    return true;
  }
  const double rho = c * sqrt_nr(g0sq);
  float Ginv[K][K], w32[K];
  const unsigned mask = (unsigned)lane + 1u;
  float F = INFINITY;
  if (mask < (1u << K)) F = cagrad_candidate32<K>(Gf, bf, (float)rho, mask, Ginv, w32);
  const int win = warp_argmin(F, lane);
  if (!(__shfl_sync(0xffffffffu, F, win) < INFINITY)) return false;
  const unsigned wm = (unsigned)win + 1u;
  const bool kin = lane < K && in_mask<K>(wm, lane);
  double w = 0.0;  // w_k on lane k
  if (__popc(wm) == 1) {
    w = kin ? 1.0 : 0.0;
  } else {
    // m = Ginv 1_S and n = Ginv b_S from the winner (fp32), on every lane
    float m[K], n[K];
#pragma unroll
    for (int ii = 0; ii < K; ++ii) {
      float mi = 0.0f, ni = 0.0f;
#pragma unroll
      for (int jj = 0; jj < K; ++jj)
        if (in_mask<K>(wm, jj)) {
          mi += Ginv[ii][jj];
          ni = fmaf(Ginv[ii][jj], bf[jj], ni);
        }
      m[ii] = __shfl_sync(0xffffffffu, mi, win);
      n[ii] = __shfl_sync(0xffffffffu, ni, win);
    }
    float mj = 0.0f, nj = 0.0f, mi_ = 0.0f, ni_ = 0.0f;
#pragma unroll
    for (int cc = 0; cc < K; ++cc) {
      if (j == cc) {
        mj = m[cc];
        nj = n[cc];
      }
      if (i == cc) {
        mi_ = m[cc];
        ni_ = n[cc];
      }
    }
    // residuals of rows i in S (1 - (G m)_i, b_i - (G n)_i); -m_i, -n_i outside
    const bool iin = i < K && in_mask<K>(wm, i);
    const double g = (j < K && in_mask<K>(wm, j)) ? gij : 0.0;
    double pm = g * (double)mj, pn = g * (double)nj;
    pm += __shfl_xor_sync(0xffffffffu, pm, 1);
    pn += __shfl_xor_sync(0xffffffffu, pn, 1);
    pm += __shfl_xor_sync(0xffffffffu, pm, 2);
    pn += __shfl_xor_sync(0xffffffffu, pn, 2);
    const float rmf = (float)(iin ? 1.0 - pm : -(double)mi_);
    const float rnf = (float)(iin ? bi - pn : -(double)ni_);
    float rm[K], rn[K];
#pragma unroll
    for (int cc = 0; cc < K; ++cc) {
      rm[cc] = __shfl_sync(0xffffffffu, rmf, 4 * cc);
      rn[cc] = __shfl_sync(0xffffffffu, rnf, 4 * cc);
    }
    // the correction through the winner's inverse; m_k, n_k in fp64 on lane k
    float mk = 0.0f, nk = 0.0f, dmk = 0.0f, dnk = 0.0f;
#pragma unroll
    for (int cc = 0; cc < K; ++cc) {
      float dm = 0.0f, dn = 0.0f;
#pragma unroll
      for (int jj = 0; jj < K; ++jj) {
        dm = fmaf(Ginv[cc][jj], rm[jj], dm);
        dn = fmaf(Ginv[cc][jj], rn[jj], dn);
      }
      dm = __shfl_sync(0xffffffffu, dm, win);
      dn = __shfl_sync(0xffffffffu, dn, win);
      if (lane == cc) {
        mk = m[cc];
        nk = n[cc];
        dmk = dm;
        dnk = dn;
      }
    }
    double bk = 0.0;
#pragma unroll
    for (int cc = 0; cc < K; ++cc)
      if (lane == cc) bk = b[cc];
    const double md = (double)mk + (double)dmk, nd = (double)nk + (double)dnk;
    double om = kin ? md : 0.0, on = kin ? nd : 0.0, nb = kin ? nd * bk : 0.0;
    om += __shfl_xor_sync(0xffffffffu, om, 1);
    on += __shfl_xor_sync(0xffffffffu, on, 1);
    nb += __shfl_xor_sync(0xffffffffu, nb, 1);
    om += __shfl_xor_sync(0xffffffffu, om, 2);
    on += __shfl_xor_sync(0xffffffffu, on, 2);
    nb += __shfl_xor_sync(0xffffffffu, nb, 2);
    om = __shfl_sync(0xffffffffu, om, 0);
    on = __shfl_sync(0xffffffffu, on, 0);
    nb = __shfl_sync(0xffffffffu, nb, 0);
    const double D = on * on - om * (nb - rho * rho);
    if (!(D > 0.0) || !(om > 0.0)) return false;
    const double sd = sqrt_nr(D);
    double u = kin ? fma(on + sd, md, -om * nd) : 0.0;
    u = u > 0.0 ? u : 0.0;
    double su = u;
    su += __shfl_xor_sync(0xffffffffu, su, 1);
    su += __shfl_xor_sync(0xffffffffu, su, 2);
    su = __shfl_sync(0xffffffffu, su, 0);
    if (!(su > 0.0)) return false;
    w = div_nr(u, su);
  }
  // optimality of the dual: grad_k = b_k + rho (G w)_k / ||g_w|| >= w^T grad
  // (equality on the support); fp32 with a margin, fp64 when marginal
  const float wf_mine = (float)w;
  float wf[K];
#pragma unroll
  for (int k = 0; k < K; ++k) wf[k] = __shfl_sync(0xffffffffu, wf_mine, k);
  {
    float v32[K], q32 = 0.0f;
#pragma unroll
    for (int k = 0; k < K; ++k) {
      float t = 0.0f;
#pragma unroll
      for (int jj = 0; jj < K; ++jj) t = fmaf(Gf[k * K + jj], wf[jj], t);
      v32[k] = t;
      q32 = fmaf(wf[k], t, q32);
    }
    if (!(q32 > 1e-12f)) return false;
    const float f32 = (float)rho / sqrtf(q32);
    float lam32 = 0.0f, g32[K];
#pragma unroll
    for (int k = 0; k < K; ++k) {
      g32[k] = fmaf(f32, v32[k], bf[k]);
      lam32 = fmaf(wf[k], g32[k], lam32);
    }
    bool clear = true;
#pragma unroll
    for (int k = 0; k < K; ++k)
      if (!in_mask<K>(wm, k) && !(g32[k] - lam32 >= 1e-5f)) clear = false;
    if (!clear) {
      double wd[K], v[K], qq = 0.0;
#pragma unroll
      for (int k = 0; k < K; ++k) wd[k] = __shfl_sync(0xffffffffu, w, k);
#pragma unroll
      for (int k = 0; k < K; ++k) {
        double t = 0.0;
#pragma unroll
        for (int jj = 0; jj < K; ++jj) t = fma(G[k * K + jj], wd[jj], t);
        v[k] = t;
        qq = fma(wd[k], t, qq);
      }
      if (!(qq > 1e-24)) return false;
      const double fd = div_nr(rho, sqrt_nr(qq));
      double lam = 0.0, gmin = 1e300;
#pragma unroll
      for (int k = 0; k < K; ++k) {
        const double gk = fma(fd, v[k], b[k]);
        lam = fma(wd[k], gk, lam);
        gmin = fmin(gmin, gk);
      }
      if (!(gmin >= lam - 1e-11)) return false;
    }
  }
  // beta = 1/K + rho w / ||g_w||, ||g_w||^2 = w^T G w in fp64 (lane (i, j):
  // w_i G_ij w_j, then a butterfly over the 16 lanes)
  const double wi = __shfl_sync(0xffffffffu, w, i & 31);
  const double wj = __shfl_sync(0xffffffffu, w, j);
  double q = (i < K && j < K) ? gij * wi * wj : 0.0;
  q += __shfl_xor_sync(0xffffffffu, q, 1);
  q += __shfl_xor_sync(0xffffffffu, q, 2);
  q += __shfl_xor_sync(0xffffffffu, q, 4);
  q += __shfl_xor_sync(0xffffffffu, q, 8);
  q = __shfl_sync(0xffffffffu, q, 0);
  if (!(q > 1e-24)) return false;
  const double f = div_nr(rho, sqrt_nr(q));
  if (lane < K) beta_out[lane] = fma(f, w, 1.0 / K);
  return true;
}

// PCGrad with one lane per task t < K (fp64): lane t runs the projections of
// its running d_t in t's order; beta_j = sum_t C_tj by a fixed shuffle tree.
template <int K>
__device__ void pcgrad_fast(const double* G, uint64_t seed, uint64_t step, int64_t b, int lane,
                            double* beta_out) {
  double r[K];
#pragma unroll
  for (int k = 0; k < K; ++k) r[k] = (k == lane) ? 1.0 : 0.0;
  if (lane < K) {
    int order[kMaxK];
    task_order(seed, step, b, K, lane, order);
#pragma unroll
    for (int q = 0; q < K - 1; ++q) {
      const int j = order[q];
      double p0 = 0.0, p1 = 0.0;
#pragma unroll
      for (int m = 0; m < K; m += 2) {
        p0 = fma(r[m], G[m * K + j], p0);
        if (m + 1 < K) p1 = fma(r[m + 1], G[(m + 1) * K + j], p1);
      }
      const double pr = p0 + p1, gjj = G[j * K + j];
      if (pr < 0.0 && gjj > 0.0) {
        const double delta = div_nr(pr, gjj);
#pragma unroll
        for (int m = 0; m < K; ++m)
          if (m == j) r[m] -= delta;
      }
    }
  }
#pragma unroll
  for (int k = 0; k < K; ++k) {
    double x = lane < K ? r[k] : 0.0;
    x += __shfl_down_sync(0xffffffffu, x, 16);
    x += __shfl_down_sync(0xffffffffu, x, 8);
    x += __shfl_down_sync(0xffffffffu, x, 4);
    x += __shfl_down_sync(0xffffffffu, x, 2);
    x += __shfl_down_sync(0xffffffffu, x, 1);
    if (lane == 0) beta_out[k] = x;
  }
}

// ---------------------------------------------------------------------------
// K >= 6: Wolfe's algorithm in fp32 with a lane-parallel Gauss-Jordan
// ---------------------------------------------------------------------------

constexpr int kUnk = kMaxK + 1;   // up to kMaxK + 1 unknowns
constexpr int kCols = kUnk + 2;   // two right-hand sides in slots kUnk, kUnk + 1

// Position of the n-th (0-based) set bit of m.
__device__ __forceinline__ int nth_set(unsigned m, int n) {
  for (int i = 0; i < n; ++i) m &= m - 1u;
  return __ffs(m) - 1;
}

__device__ __forceinline__ int warp_argmin_f(float val, int lane) { return warp_argmin(val, lane); }

__device__ __forceinline__ float warp_sum_f(float x) {
  for (int off = 16; off > 0; off >>= 1) x += __shfl_xor_sync(0xffffffffu, x, off);
  return x;
}

// Lane i < m holds row i of an m-unknown system: coefficients in row[0..m-1]
// (slots m .. kUnk-1 are zero) and two right-hand sides in row[kUnk] and
// row[kUnk + 1].  Gauss-Jordan with partial pivoting across lanes;
// afterwards lane i < m holds the two solutions' i-th entries in the same
// slots.  False when a pivot is below `piv`.
__device__ bool warp_gauss_jordan(float (&row)[kCols], int m, int lane, float piv) {
  bool ok = true;
#pragma unroll
  for (int c = 0; c < kUnk; ++c) {
    if (c >= m) break;
    float a = (lane >= c && lane < m) ? fabsf(row[c]) : -1.0f;
    int p = lane;
    for (int off = 16; off > 0; off >>= 1) {
      const float a2 = __shfl_xor_sync(0xffffffffu, a, off);
      const int p2 = __shfl_xor_sync(0xffffffffu, p, off);
      if (a2 > a || (a2 == a && p2 < p)) {
        a = a2;
        p = p2;
      }
    }
    if (!(a > piv)) ok = false;
    const int src = lane == c ? p : (lane == p ? c : lane);
#pragma unroll
    for (int j = c; j < kCols; ++j) row[j] = __shfl_sync(0xffffffffu, row[j], src);
    const float inv = __frcp_rn(__shfl_sync(0xffffffffu, row[c], c));
    const float f = row[c];
#pragma unroll
    for (int j = c; j < kCols; ++j) {
      const float pj = __shfl_sync(0xffffffffu, row[j], c) * inv;
      if (lane == c) row[j] = pj;
      else if (lane < m) row[j] = fmaf(-f, pj, row[j]);
    }
  }
  return ok;
}

// Bordered system of the affine minimum-norm point of support smask
// (s = |S| rows of G_SS | 1, then the row 1^T | 0); rhs supplied per lane.
__device__ __forceinline__ void mgda_rows(const float* Gf, int K, unsigned smask, int lane,
                                          float rhs, float (&row)[kCols]) {
  const int s = __popc(smask);
  const int pi = lane < s ? nth_set(smask, lane) : 0;
#pragma unroll
  for (int j = 0; j < kUnk; ++j) {
    float v = 0.0f;
    if (j < s) {
      const int pj = nth_set(smask, j);
      v = lane < s ? Gf[pi * K + pj] : (lane == s ? 1.0f : 0.0f);
    } else if (j == s) {
      v = lane < s ? 1.0f : 0.0f;
    }
    row[j] = v;
  }
  row[kUnk] = rhs;
  row[kUnk + 1] = 0.0f;
}

// Exact MGDA for any K (used for K >= 6): Wolfe's minimum-norm-point method
// on the fp32 Gram with lane k holding weight lam_k, then one fp64
// refinement of the final support and the optimality check.  False (beta
// untouched) if a system is singular or the check fails.
__device__ bool mgda_wolfe_warp(int K, const double* G, const float* Gf, int lane,
                                double* beta_out) {
  const bool act = lane < K;
  const int k0 = warp_argmin_f(act ? Gf[lane * K + lane] : INFINITY, lane);
  bool in = lane == k0;
  float lam = in ? 1.0f : 0.0f;
  float row[kCols];
  for (int major = 0; major < 4 * K + 4; ++major) {
    float v = 0.0f;
    for (int j = 0; j < K; ++j) {
      const float lj = __shfl_sync(0xffffffffu, lam, j);
      if (act) v = fmaf(Gf[lane * K + j], lj, v);
    }
    const float xx = warp_sum_f(act ? lam * v : 0.0f);
    const int jn = warp_argmin_f(act ? v : INFINITY, lane);
    const float vj = __shfl_sync(0xffffffffu, v, jn);
    if (vj >= xx - 1e-6f) break;
    if (__shfl_sync(0xffffffffu, in ? 1 : 0, jn)) break;
    if (lane == jn) {
      in = true;
      lam = 0.0f;
    }
    bool settled = false;
    for (int minor = 0; minor <= K + 1 && !settled; ++minor) {
      const unsigned smask = __ballot_sync(0xffffffffu, in && act);
      const int s = __popc(smask);
      if (s == 0) return false;
      mgda_rows(Gf, K, smask, lane, lane == s ? 1.0f : 0.0f, row);
      if (!warp_gauss_jordan(row, s + 1, lane, 1e-6f)) return false;
      const int rank = __popc(smask & ((1u << lane) - 1u));
      const float mu_all = __shfl_sync(0xffffffffu, row[kUnk], in ? rank : 0);
      const float mu = in ? mu_all : 0.0f;
      if (__all_sync(0xffffffffu, !in || mu > 1e-7f)) {
        lam = mu;
        settled = true;
        break;
      }
      const float t = (in && mu <= 1e-7f) ? ((lam - mu) > 0.0f ? lam / (lam - mu) : 0.0f)
                                          : INFINITY;
      const int drop = warp_argmin_f(t, lane);
      const float theta = __shfl_sync(0xffffffffu, t, drop);
      lam = in ? (1.0f - theta) * lam + theta * mu : 0.0f;
      if (lane == drop || lam <= 1e-7f) {
        in = false;
        lam = 0.0f;
      }
    }
    if (!settled) return false;
  }
  // one fp64 refinement of the final support's bordered system
  const unsigned smask = __ballot_sync(0xffffffffu, in && act);
  const int s = __popc(smask);
  if (s == 0) return false;
  mgda_rows(Gf, K, smask, lane, lane == s ? 1.0f : 0.0f, row);
  if (!warp_gauss_jordan(row, s + 1, lane, 1e-6f)) return false;
  double z = (lane <= s) ? (double)row[kUnk] : 0.0;   // lane i <= s: unknown i
  double r = 0.0;
  {
    const int pi = lane < s ? nth_set(smask, lane) : 0;
    double acc = 0.0;
    for (int j = 0; j <= s; ++j) {
      const double zj = __shfl_sync(0xffffffffu, z, j);
      if (lane < s) {
        const double a = j < s ? G[pi * K + nth_set(smask, j)] : 1.0;
        acc = fma(a, zj, acc);
      } else if (lane == s && j < s) {
        acc += zj;
      }
    }
    r = lane < s ? -acc : (lane == s ? 1.0 - acc : 0.0);
  }
  mgda_rows(Gf, K, smask, lane, (float)r, row);
  if (!warp_gauss_jordan(row, s + 1, lane, 1e-6f)) return false;
  z += (lane <= s) ? (double)row[kUnk] : 0.0;
  // alpha on lanes k < K
  const int rank = __popc(smask & ((1u << lane) - 1u));
  const bool ink = act && ((smask >> lane) & 1u);
  const double zk = __shfl_sync(0xffffffffu, z, ink ? rank : 0);
  double alpha = (ink && zk > 0.0) ? zk : 0.0;
  double sum = alpha;
  for (int off = 16; off > 0; off >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, off);
  alpha *= (2.0 - sum);
  // optimality (proof of Theorem 3.1): fp32 with a margin, fp64 if marginal
  const float a32 = (float)alpha;
  float v32 = 0.0f;
  for (int j = 0; j < K; ++j) {
    const float aj = __shfl_sync(0xffffffffu, a32, j);
    if (act) v32 = fmaf(Gf[lane * K + j], aj, v32);
  }
  const float xx32 = warp_sum_f(act ? a32 * v32 : 0.0f);
  const bool clear = !act || ink || (v32 - xx32 >= 1e-5f);
  if (!__all_sync(0xffffffffu, clear)) {
    double v = 0.0;
    for (int j = 0; j < K; ++j) {
      const double aj = __shfl_sync(0xffffffffu, alpha, j);
      if (act) v = fma(G[lane * K + j], aj, v);
    }
    double xx = act ? alpha * v : 0.0;
    for (int off = 16; off > 0; off >>= 1) xx += __shfl_xor_sync(0xffffffffu, xx, off);
    if (!__all_sync(0xffffffffu, !act || v >= xx - kKkt)) return false;
  }
  if (act) beta_out[lane] = alpha;
  return true;
}

// Rows of G_SS [m n] = [1 b_S] for support smask (lane i < s: row i).
__device__ __forceinline__ void cagrad_rows(const float* Gf, int K, unsigned smask, int lane,
                                            float bi, float r1, float r2, float (&row)[kCols]) {
  const int s = __popc(smask);
  const int pi = lane < s ? nth_set(smask, lane) : 0;
#pragma unroll
  for (int j = 0; j < kUnk; ++j)
    row[j] = (j < s && lane < s) ? Gf[pi * K + nth_set(smask, j)] : 0.0f;
  row[kUnk] = lane < s ? r1 : 0.0f;
  row[kUnk + 1] = lane < s ? r2 : 0.0f;
  (void)bi;
}

// Exact CAGrad for any K (used for K >= 6): active-set method on the dual
// min_{w in simplex} b^T w + rho ||g_w|| from the best vertex, with the
// closed-form stationary point of each support (see cag_affine) solved by
// the lane-parallel Gauss-Jordan in fp32; then m, n refined once in fp64,
// the closed form in fp64 and the optimality check.  Lane k holds w_k.
__device__ bool cagrad_active_warp(int K, const double* G, const float* Gf, double c, int lane,
                                   double* beta_out) {
  const bool act = lane < K;
  // b_k = <g_k, g0>, ||g0||^2 (fp64 for the final coefficients)
  double bd = 0.0;
  if (act)
    for (int j = 0; j < K; ++j) bd += G[lane * K + j];
  double tot = bd;
  for (int off = 16; off > 0; off >>= 1) tot += __shfl_xor_sync(0xffffffffu, tot, off);
  bd *= 1.0 / K;
  const double g0sq = tot * (1.0 / ((double)K * K));
  if (!(c > 0.0) || !(g0sq > 0.0)) {
    if (act) beta_out[lane] = 1.0 / K;
    return true;
  }
  // (no sign condition on b: the final optimality check certifies the
  // result, see cagrad_fast)
  const double rho = c * sqrt_nr(g0sq);
  const float rhof = (float)rho, bf = (float)bd;
  const float Fv = act ? bf + rhof * sqrtf(fmaxf(Gf[lane * K + lane], 0.0f)) : INFINITY;
  const int k0 = warp_argmin_f(Fv, lane);
  bool in = lane == k0;
  float w = in ? 1.0f : 0.0f;
  float row[kCols];
  for (int major = 0; major < 4 * K + 4; ++major) {
    float v = 0.0f;
    for (int j = 0; j < K; ++j) {
      const float wj = __shfl_sync(0xffffffffu, w, j);
      if (act) v = fmaf(Gf[lane * K + j], wj, v);
    }
    const float q = warp_sum_f(act ? w * v : 0.0f);
    if (!(q > 1e-20f)) return false;
    const float gk = act ? bf + rhof * v / sqrtf(q) : INFINITY;
    const float lam = warp_sum_f(act ? w * gk : 0.0f);
    const int jn = warp_argmin_f(gk, lane);
    if (__shfl_sync(0xffffffffu, gk, jn) >= lam - 1e-6f) break;
    if (__shfl_sync(0xffffffffu, in ? 1 : 0, jn)) break;
    if (lane == jn) {
      in = true;
      w = 0.0f;
    }
    bool settled = false;
    for (int minor = 0; minor <= K + 1 && !settled; ++minor) {
      const unsigned smask = __ballot_sync(0xffffffffu, in && act);
      const int s = __popc(smask);
      if (s == 0) return false;
      const int pi = lane < s ? nth_set(smask, lane) : 0;
      cagrad_rows(Gf, K, smask, lane, 0.0f, 1.0f, __shfl_sync(0xffffffffu, bf, pi), row);
      if (!warp_gauss_jordan(row, s, lane, 1e-6f)) return false;
      const float mi = lane < s ? row[kUnk] : 0.0f, ni = lane < s ? row[kUnk + 1] : 0.0f;
      const float bpi = __shfl_sync(0xffffffffu, bf, pi);
      const float om = warp_sum_f(mi), on = warp_sum_f(ni), nb = warp_sum_f(lane < s ? ni * bpi : 0.0f);
      const float D = on * on - om * (nb - rhof * rhof);
      if (!(om > 0.0f) || !(D > 0.0f)) return false;
      const float sd = sqrtf(D), lamc = (on + sd) / om;
      const float zi = (lamc * mi - ni) / sd;                  // lane i < s: support entry i
      const int rank = __popc(smask & ((1u << lane) - 1u));
      const float zk_all = __shfl_sync(0xffffffffu, zi, in ? rank : 0);
      const float z = in ? zk_all : 0.0f;
      if (__all_sync(0xffffffffu, !in || z > 1e-7f)) {
        const float zs = warp_sum_f(z);
        w = z / zs;
        settled = true;
        break;
      }
      const float t = (in && z <= 1e-7f) ? ((w - z) > 0.0f ? w / (w - z) : 0.0f) : INFINITY;
      const int drop = warp_argmin_f(t, lane);
      const float theta = __shfl_sync(0xffffffffu, t, drop);
      w = in ? (1.0f - theta) * w + theta * z : 0.0f;
      if (lane == drop || w <= 1e-7f) {
        in = false;
        w = 0.0f;
      }
    }
    if (!settled) return false;
  }
  // fp64: m = G_SS^-1 1 and n = G_SS^-1 b_S with one refinement step
  const unsigned smask = __ballot_sync(0xffffffffu, in && act);
  const int s = __popc(smask);
  if (s == 0) return false;
  const int pi = lane < s ? nth_set(smask, lane) : 0;
  const double bpi = __shfl_sync(0xffffffffu, bd, pi);
  cagrad_rows(Gf, K, smask, lane, 0.0f, 1.0f, (float)bpi, row);
  if (!warp_gauss_jordan(row, s, lane, 1e-6f)) return false;
  double md = lane < s ? (double)row[kUnk] : 0.0, nd = lane < s ? (double)row[kUnk + 1] : 0.0;
  double rm = 0.0, rn = 0.0;
  {
    double am = 0.0, an = 0.0;
    for (int j = 0; j < s; ++j) {
      const double mj = __shfl_sync(0xffffffffu, md, j), nj = __shfl_sync(0xffffffffu, nd, j);
      if (lane < s) {
        const double a = G[pi * K + nth_set(smask, j)];
        am = fma(a, mj, am);
        an = fma(a, nj, an);
      }
    }
    rm = lane < s ? 1.0 - am : 0.0;
    rn = lane < s ? bpi - an : 0.0;
  }
  cagrad_rows(Gf, K, smask, lane, 0.0f, (float)rm, (float)rn, row);
  if (!warp_gauss_jordan(row, s, lane, 1e-6f)) return false;
  if (lane < s) {
    md += (double)row[kUnk];
    nd += (double)row[kUnk + 1];
  }
  double om = md, on = nd, nb = lane < s ? nd * bpi : 0.0;
  for (int off = 16; off > 0; off >>= 1) {
    om += __shfl_xor_sync(0xffffffffu, om, off);
    on += __shfl_xor_sync(0xffffffffu, on, off);
    nb += __shfl_xor_sync(0xffffffffu, nb, off);
  }
  const double D = on * on - om * (nb - rho * rho);
  if (!(om > 0.0) || !(D > 0.0)) return false;
  const double sd = sqrt_nr(D), lamc = div_nr(on + sd, om), isd = div_nr(1.0, sd);
  const double zi = lane < s ? (lamc * md - nd) * isd : 0.0;
  const int rank = __popc(smask & ((1u << lane) - 1u));
  const bool ink = act && ((smask >> lane) & 1u);
  const double zk = __shfl_sync(0xffffffffu, zi, ink ? rank : 0);
  double wd = (ink && zk > 0.0) ? zk : 0.0;
  double sum = wd;
  for (int off = 16; off > 0; off >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, off);
  wd *= (2.0 - sum);
  // optimality of the dual (fp32 with a margin, fp64 if marginal), and
  // beta = 1/K + rho w / ||g_w|| with ||g_w|| in fp64
  double vd = 0.0;
  for (int j = 0; j < K; ++j) {
    const double wj = __shfl_sync(0xffffffffu, wd, j);
    if (act) vd = fma(G[lane * K + j], wj, vd);
  }
  double qd = act ? wd * vd : 0.0;
  for (int off = 16; off > 0; off >>= 1) qd += __shfl_xor_sync(0xffffffffu, qd, off);
  if (!(qd > 1e-24)) return false;
  const double f = div_nr(rho, sqrt_nr(qd));
  const double gk = act ? fma(f, vd, bd) : 1e300;
  double lam = act ? wd * gk : 0.0;
  for (int off = 16; off > 0; off >>= 1) lam += __shfl_xor_sync(0xffffffffu, lam, off);
  if (!__all_sync(0xffffffffu, !act || ink || gk >= lam - 1e-11)) return false;
  if (act) beta_out[lane] = fma(f, wd, 1.0 / K);
  return true;
}

// Large-K (K > kEnumMaxK) MGDA and CAGrad: one copy of the lane-parallel
// active-set solvers per kernel, whatever the number of K cases around it.
__device__ bool solve_large(int K, int rule, const double* G, const float* Gf,
                            const SolveParams& p, int lane, double* beta_out) {
  if (!(p.flags & BKMOO_FLAG_POLISH)) return false;
  if (rule == BKMOO_MGDA) return mgda_wolfe_warp(K, G, Gf, lane, beta_out);
  if (rule == BKMOO_CAGRAD) return cagrad_active_warp(K, G, Gf, p.cagrad_c, lane, beta_out);
  return false;
}

// kLarge: whether this instantiation carries the large-K solvers itself
// (the runtime-K dispatch below calls solve_large once, outside its switch).
template <int K, bool kLarge>
__device__ bool solve_fast_k(int rule, const double* G, const float* Gf, const SolveParams& p,
                             int64_t b, int lane, double* beta_out) {
  if (rule == BKMOO_PCGRAD) {
    pcgrad_fast<K>(G, p.seed, p.step, b, lane, beta_out);
    return true;
  }
  if (!(p.flags & BKMOO_FLAG_POLISH)) return false;
  if (K > kEnumMaxK) return kLarge ? solve_large(K, rule, G, Gf, p, lane, beta_out) : false;
  if (rule == BKMOO_MGDA) {
    if (K < 2 || (K == 2 && (p.flags & BKMOO_FLAG_CLOSED_FORM_K2))) return false;
    return mgda_fast<(K <= kEnumMaxK ? K : 2)>(G, Gf, lane, beta_out);
  }
  if (rule == BKMOO_CAGRAD) {
    constexpr int KE = K <= kEnumMaxK ? K : 1;
    if constexpr (KE <= 4)
      return cagrad_fast_warp<KE>(G, Gf, p.cagrad_c, lane, beta_out);
    else
      return cagrad_fast<KE>(G, Gf, p.cagrad_c, lane, beta_out);
  }
  return false;
}

// Dispatch on K; true when a fast path produced beta (valid on every lane
// after the caller's __syncwarp).
__device__ bool solve_fast(int K, int rule, const double* G, const float* Gf,
                           const SolveParams& p, int64_t b, int lane, double* beta_out) {
  if (K > kEnumMaxK && rule != BKMOO_PCGRAD) return solve_large(K, rule, G, Gf, p, lane, beta_out);
  switch (K) {
#define BKMOO_FAST_CASE(k) \
  case k: return solve_fast_k<k, false>(rule, G, Gf, p, b, lane, beta_out);
    BKMOO_FAST_CASE(1) BKMOO_FAST_CASE(2) BKMOO_FAST_CASE(3) BKMOO_FAST_CASE(4)
    BKMOO_FAST_CASE(5) BKMOO_FAST_CASE(6) BKMOO_FAST_CASE(7) BKMOO_FAST_CASE(8)
    BKMOO_FAST_CASE(9) BKMOO_FAST_CASE(10) BKMOO_FAST_CASE(11) BKMOO_FAST_CASE(12)
    BKMOO_FAST_CASE(13) BKMOO_FAST_CASE(14) BKMOO_FAST_CASE(15) BKMOO_FAST_CASE(16)
#undef BKMOO_FAST_CASE
    default: return false;
  }
}

// ---------------------------------------------------------------------------
// per bucket (whole warp)
// ---------------------------------------------------------------------------

// The whole warp enters with G (K x K) in shared memory; G is normalised in
// place.  beta_out (shared, K entries) and the returned status are valid on
// every lane after the call.
// KC > 0: K is the compile-time constant KC (one solver instantiation);
// KC = 0: K is a runtime value dispatched over 1..kMaxK.
template <int KC>
__device__ int solve_bucket_warp(int K, double* G, float* Gf, const SolveParams& p, int64_t b,
                                 double* beta_out, int lane) {
  // finiteness and the largest diagonal entry from the bit patterns
  // (non-negative doubles order as integers), then an exact power-of-two
  // scaling that brings max_k G_kk into [1, 2)
  bool finite = true;
  long long dmax = 0;
  for (int i = lane; i < K * K; i += 32) {
    const long long bits = __double_as_longlong(G[i]);
    if (((bits >> 52) & 0x7ff) == 0x7ff) finite = false;
    if (i / K == i % K && bits > dmax) dmax = bits;
  }
  finite = __all_sync(0xffffffffu, finite);
  for (int off = 16; off > 0; off >>= 1) {
    const long long o = __shfl_xor_sync(0xffffffffu, dmax, off);
    dmax = o > dmax ? o : dmax;
  }
  if (!finite) {
    if (lane == 0)
      for (int k = 0; k < K; ++k) beta_out[k] = 1.0 / K;
    __syncwarp();
    return BKMOO_ERR_NONFINITE;
  }
  double top = 1.0;
  if (dmax > 0) {
    const int e = (int)((dmax >> 52) & 0x7ff) - 1023;
    if (e > -1022 && e < 1023) {
      const double f = __longlong_as_double((long long)(1023 - e) << 52);
      for (int i = lane; i < K * K; i += 32) G[i] *= f;
      top = __longlong_as_double(dmax) * f;
    } else {  // extreme scales: plain division
      const double inv = 1.0 / __longlong_as_double(dmax);
      for (int i = lane; i < K * K; i += 32) G[i] *= inv;
    }
  }
  __syncwarp();
  for (int i = lane; i < K * K; i += 32) Gf[i] = (float)G[i];
  __syncwarp();
  SolveParams q = p;
  q.tol = p.tol * top;  // the stopping test is relative to max_k G_kk
  int st = BKMOO_OK;
  bool fast;
  if constexpr (KC > 0)
    fast = solve_fast_k<KC, true>(q.rule, G, Gf, q, b, lane, beta_out);
  else
    fast = solve_fast(K, q.rule, G, Gf, q, b, lane, beta_out);
  if (!fast && lane == 0) {
    double beta[kMaxK];
    switch (q.rule) {
      case BKMOO_MGDA: st = solve_mgda(K, G, q, beta); break;
      case BKMOO_PCGRAD: st = solve_pcgrad(K, G, q, b, beta); break;
      case BKMOO_CAGRAD: st = solve_cagrad(K, G, q, beta); break;
      default:
        for (int k = 0; k < K; ++k) beta[k] = 1.0 / K;
    }
    for (int k = 0; k < K; ++k) beta_out[k] = beta[k];
  }
  st = __shfl_sync(0xffffffffu, st, 0);
  __syncwarp();
  return st;
}

}  // namespace
}  // namespace solver
}  // namespace bkmoo
