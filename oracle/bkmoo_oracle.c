/*
 * bkmoo_oracle.c -- plain, slow, fp64 CPU oracle for Bucket-Level MOO
 * ("Multilingual Fine-Tuning via Localized Gradient Conflict Resolution",
 * arXiv 2606.05613).
 *
 * TEST INFRASTRUCTURE.  Only the test-suite, the smoke check and the
 * benchmark's CPU-baseline leg load this library.  It shares no code, header,
 * table or constant generator with the CUDA library, and neither calls the
 * other.
 *
 * Notation.  K = number of languages (the paper's T), B = number of parameter
 * buckets (the paper's K), G = the K x K Gram matrix of one bucket,
 * G[i][j] = <g_i, g_j> restricted to the bucket.
 *
 * Every input element is read exactly as stored (fp32, or bf16 widened
 * exactly) and every operation is done in double precision, one bucket at a
 * time, in plain sequential order.  The only parallelism is an optional
 * OpenMP loop over independent buckets in bko_resolve(); it does not change
 * any bucket's arithmetic.
 *
 * Parity status.  The bucket rule R1 (bko_plan), the PCGrad order generator
 * (bko_pcgrad_order), the Frank-Wolfe initialisation and tie-breaks
 * (bko_mgda_fw) and the non-finite policy are definitions of this library:
 * the paper fixes none of them.  They are "parity unpinned" beyond the
 * properties the tests check (valid partitions, valid permutations, FW
 * reducing to the K=2 closed form, descent of the objective).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define BKO_F32 0
#define BKO_BF16 1

#define BKO_MGDA 0
#define BKO_PCGRAD 1
#define BKO_CAGRAD 2
#define BKO_MEAN 3

#define BKO_MGDA_EXACT 0 /* Wolfe minimum-norm point (K=2: closed form)  */
#define BKO_MGDA_FW 1    /* Frank-Wolfe replay with a capped iteration count */
#define BKO_MGDA_ENUM 2  /* enumeration of every support (K <= 16)      */

#define BKO_OK 0
#define BKO_NONFINITE 3

#define KMAX 16

typedef struct {
  int32_t mgda_mode;  /* BKO_MGDA_* */
  int32_t max_iter;   /* Frank-Wolfe iterations for BKO_MGDA_FW */
  double tol;         /* relative Frank-Wolfe duality-gap stop */
  double cagrad_c;    /* CAGrad conflict-aversion c in [0, 1) */
  uint64_t seed;      /* PCGrad order */
  uint64_t step;      /* PCGrad order */
} bko_params;

/* ------------------------------------------------------------------------ */
/* element access                                                            */
/* ------------------------------------------------------------------------ */

static double load_elem(const void* base, int32_t dtype, int64_t i) {
  if (dtype == BKO_F32) return (double)((const float*)base)[i];
  /* bf16 is the upper half of an IEEE binary32: widening is exact. */
  uint32_t u = (uint32_t)((const uint16_t*)base)[i] << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return (double)f;
}

/* ------------------------------------------------------------------------ */
/* Bucket partition (Section 3.2, Figure 4 caption; Algorithm 1 input).      */
/* ------------------------------------------------------------------------ */

/*
 * Rule R1.  The paper fills fixed-size buckets sequentially during the
 * backward pass, starting from the last parameters (Figure 4 caption).  So
 * the flat per-language gradient lists the tensors in REVERSE registration
 * order, and a bucket holds at most cap = floor(bucket_bytes / elem_bytes)
 * elements.  Walking that list: a tensor that does not fit in the open bucket
 * closes it first; a tensor larger than cap is split into cap-sized pieces;
 * what remains joins the open bucket.  On a single tensor this is plain
 * fixed-size chunking.  Empty tensors are skipped.
 *
 * Returns the number of buckets B (offsets[0] = 0, offsets[B] = N), -1 on
 * invalid arguments, -2 if out_offsets is non-NULL but out_cap < B + 1.
 */
int64_t bko_plan(const int64_t* sizes, int32_t n_params, int32_t elem_bytes,
                 int64_t bucket_bytes, int64_t* out_offsets, int64_t out_cap) {
  if (!sizes || n_params < 0 || elem_bytes <= 0 || bucket_bytes <= 0) return -1;
  int64_t cap = bucket_bytes / elem_bytes;
  if (cap < 1) return -1;
  for (int32_t t = 0; t < n_params; ++t)
    if (sizes[t] < 0) return -1;

  int64_t n_b = 0, pos = 0, cur = 0;
  int too_small = 0;
#define CLOSE_BUCKET()                                   \
  do {                                                   \
    ++n_b;                                               \
    if (out_offsets) {                                   \
      if (n_b + 1 > out_cap) too_small = 1;              \
      else out_offsets[n_b] = pos;                       \
    }                                                    \
  } while (0)

  if (out_offsets) {
    if (out_cap < 1) return -2;
    out_offsets[0] = 0;
  }
  for (int32_t t = n_params - 1; t >= 0; --t) {
    int64_t n = sizes[t];
    if (n == 0) continue;
    if (cur > 0 && cur + n > cap) {
      CLOSE_BUCKET();
      cur = 0;
    }
    while (n > cap) {
      pos += cap;
      CLOSE_BUCKET();
      n -= cap;
    }
    cur += n;
    pos += n;
  }
  if (cur > 0) CLOSE_BUCKET();
#undef CLOSE_BUCKET
  if (too_small) return -2;
  return n_b;
}

/* ------------------------------------------------------------------------ */
/* Gram matrix of one bucket (the inner products of Eq. 2, Eq. 6, Eq. 8).    */
/* ------------------------------------------------------------------------ */

/* G[i*K+j] = sum_{e in [begin, begin+n)} x_i[e] * x_j[e], each entry summed
 * sequentially in increasing e (one pass over the elements, every entry i <= j
 * keeping its own running sum). */
void bko_gram(int32_t K, int32_t dtype, const void* const* x, int64_t begin,
              int64_t n, double* G) {
  double s[KMAX * KMAX], v[KMAX];
  for (int32_t i = 0; i < K * K; ++i) s[i] = 0.0;
  for (int64_t e = begin; e < begin + n; ++e) {
    for (int32_t i = 0; i < K; ++i) v[i] = load_elem(x[i], dtype, e);
    for (int32_t i = 0; i < K; ++i)
      for (int32_t j = i; j < K; ++j) s[i * K + j] += v[i] * v[j];
  }
  for (int32_t i = 0; i < K; ++i)
    for (int32_t j = i; j < K; ++j) {
      G[i * K + j] = s[i * K + j];
      G[j * K + i] = s[i * K + j];
    }
}

/* ------------------------------------------------------------------------ */
/* Small dense linear algebra                                                */
/* ------------------------------------------------------------------------ */

/* Solve A y = r (m x m, row-major, both overwritten; y returned in r) by
 * Gaussian elimination with partial pivoting.  Returns 0 when a pivot is
 * below piv_tol in magnitude (treated as singular). */
static int solve_dense(int m, double* A, double* r, double piv_tol) {
  for (int c = 0; c < m; ++c) {
    int p = c;
    for (int i = c + 1; i < m; ++i)
      if (fabs(A[i * m + c]) > fabs(A[p * m + c])) p = i;
    if (!(fabs(A[p * m + c]) > piv_tol)) return 0;
    if (p != c) {
      for (int j = 0; j < m; ++j) {
        double t = A[c * m + j];
        A[c * m + j] = A[p * m + j];
        A[p * m + j] = t;
      }
      double t = r[c];
      r[c] = r[p];
      r[p] = t;
    }
    for (int i = c + 1; i < m; ++i) {
      double f = A[i * m + c] / A[c * m + c];
      if (f == 0.0) continue;
      for (int j = c; j < m; ++j) A[i * m + j] -= f * A[c * m + j];
      r[i] -= f * r[c];
    }
  }
  for (int i = m - 1; i >= 0; --i) {
    double s = r[i];
    for (int j = i + 1; j < m; ++j) s -= A[i * m + j] * r[j];
    r[i] = s / A[i * m + i];
  }
  return 1;
}

#define PIV_TOL 1e-13

/* Minimiser of ||sum_{k in S} mu_k g_k||^2 subject to sum mu = 1, with mu
 * unrestricted in sign: the stationarity system
 *   [G_SS 1; 1^T 0] [mu; nu] = [0; 1].
 * Gn is the normalised Gram (largest diagonal 1).  Returns 0 if singular. */
static int affine_min_norm(int K, const double* Gn, const int* S, int s,
                           double* mu) {
  double A[(KMAX + 1) * (KMAX + 1)], r[KMAX + 1];
  int m = s + 1;
  for (int i = 0; i < s; ++i) {
    for (int j = 0; j < s; ++j) A[i * m + j] = Gn[S[i] * K + S[j]];
    A[i * m + s] = 1.0;
    r[i] = 0.0;
  }
  for (int j = 0; j < s; ++j) A[s * m + j] = 1.0;
  A[s * m + s] = 0.0;
  r[s] = 1.0;
  if (!solve_dense(m, A, r, PIV_TOL)) return 0;
  for (int i = 0; i < s; ++i) mu[i] = r[i];
  return 1;
}

static double quad_form(int K, const double* G, const double* w) {
  double s = 0.0;
  for (int i = 0; i < K; ++i)
    for (int j = 0; j < K; ++j) s += w[i] * G[i * K + j] * w[j];
  return s;
}

/* Copy G scaled so that its largest diagonal entry is 1.  Returns the scale
 * (0 when every diagonal entry is 0, i.e. every gradient of the bucket is 0).
 * Every rule below is invariant under a positive scaling of G. */
static double normalise(int K, const double* G, double* Gn) {
  double s = 0.0;
  for (int k = 0; k < K; ++k)
    if (G[k * K + k] > s) s = G[k * K + k];
  for (int i = 0; i < K * K; ++i) Gn[i] = (s > 0.0) ? G[i] / s : 0.0;
  return s;
}

static int all_finite(int n, const double* v) {
  for (int i = 0; i < n; ++i)
    if (!isfinite(v[i])) return 0;
  return 1;
}

/* ------------------------------------------------------------------------ */
/* MGDA: min_{alpha in simplex} || sum_k alpha_k g_k ||^2  (Eq. 3; its      */
/* bucket form Eq. 6 with the simplex of Algorithm 1 and Theorem 3.1).       */
/* ------------------------------------------------------------------------ */

/* K = 2 closed form: d = gamma g_1 + (1 - gamma) g_2 with
 * gamma = clamp(<g_2 - g_1, g_2> / ||g_1 - g_2||^2, 0, 1), which is the
 * minimiser of the one-dimensional quadratic along the segment.  Identical
 * gradients (denominator 0) take gamma = 1/2; d is the same for any gamma. */
void bko_mgda_k2(const double* G, double* alpha) {
  double den = G[0] + G[3] - 2.0 * G[1];
  double gam = 0.5;
  if (den > 0.0) {
    gam = (G[3] - G[1]) / den;
    if (gam < 0.0) gam = 0.0;
    if (gam > 1.0) gam = 1.0;
  }
  alpha[0] = gam;
  alpha[1] = 1.0 - gam;
}

/*
 * Exact minimum-norm point of conv{g_1..g_K} by Wolfe's algorithm
 * (P. Wolfe, "Finding the nearest point in a polytope", Math. Programming
 * 11, 1976), written on the Gram matrix.  It keeps a corral S (an affinely
 * independent set of gradients) with weights lam on it:
 *   major cycle: x = sum lam_k g_k; if every g_j has <x, g_j> >= ||x||^2
 *     (up to 1e-13 of the largest squared norm) x is optimal (this is the
 *     inequality used in the proof of Theorem 3.1); else add the g_j of least
 *     <x, g_j>;
 *   minor cycle: y = affine minimum-norm point of S; if y lies inside the
 *     relative interior of conv S take it, else move from x towards y to the
 *     boundary and drop the gradients whose weight reached 0.
 * Returns the number of major cycles, or -1 if it stalls on a singular
 * system.
 */
int bko_mgda_wolfe(int32_t K, const double* G, double* alpha) {
  double Gn[KMAX * KMAX], v[KMAX], mu[KMAX + 1];
  int S[KMAX], s = 0;
  for (int k = 0; k < K; ++k) alpha[k] = 0.0;
  if (K == 1) {
    alpha[0] = 1.0;
    return 0;
  }
  double scale = normalise(K, G, Gn);
  int k0 = 0;
  for (int k = 1; k < K; ++k)
    if (Gn[k * K + k] < Gn[k0 * K + k0]) k0 = k;
  S[s++] = k0;
  alpha[k0] = 1.0;
  if (scale == 0.0) return 0;

  const double z1 = 1e-13, z2 = 1e-15;
  for (int major = 0; major < 50 * K; ++major) {
    double xx = 0.0;
    for (int k = 0; k < K; ++k) {
      double t = 0.0;
      for (int j = 0; j < K; ++j) t += Gn[k * K + j] * alpha[j];
      v[k] = t;
    }
    for (int k = 0; k < K; ++k) xx += alpha[k] * v[k];
    int jmin = 0;
    for (int k = 1; k < K; ++k)
      if (v[k] < v[jmin]) jmin = k;
    if (v[jmin] >= xx - z1) return major;
    for (int i = 0; i < s; ++i)
      if (S[i] == jmin) return major; /* no progress possible */
    S[s++] = jmin;
    alpha[jmin] = 0.0;

    for (int minor = 0; minor <= K + 1; ++minor) {
      if (!affine_min_norm(K, Gn, S, s, mu)) {
        /* drop the point just added and stop */
        alpha[jmin] = 0.0;
        return -1;
      }
      int inside = 1;
      for (int i = 0; i < s; ++i)
        if (!(mu[i] > z2)) inside = 0;
      if (inside) {
        for (int i = 0; i < s; ++i) alpha[S[i]] = mu[i];
        break;
      }
      double theta = 1.0;
      int drop = -1;
      for (int i = 0; i < s; ++i) {
        if (mu[i] <= z2) {
          double a = alpha[S[i]];
          double den = a - mu[i];
          double t = den > 0.0 ? a / den : 0.0;
          if (drop < 0 || t < theta) {
            theta = t;
            drop = i;
          }
        }
      }
      for (int i = 0; i < s; ++i)
        alpha[S[i]] = (1.0 - theta) * alpha[S[i]] + theta * mu[i];
      alpha[S[drop]] = 0.0;
      int w = 0;
      for (int i = 0; i < s; ++i)
        if (alpha[S[i]] > z2) S[w++] = S[i];
        else alpha[S[i]] = 0.0;
      s = w;
    }
  }
  return 50 * K;
}

/*
 * Exact minimum-norm point by enumerating every support S (independent of
 * Wolfe's algorithm; used to pin it).  The minimiser lies in the relative
 * interior of conv S for some affinely independent S, where it is the affine
 * minimum-norm point of S; every feasible affine minimiser is a feasible
 * point, so the least objective among them is the minimum.  Cost 2^K linear
 * solves: meant for small K and few buckets.
 */
void bko_mgda_enum(int32_t K, const double* G, double* alpha) {
  double Gn[KMAX * KMAX], mu[KMAX + 1], w[KMAX];
  int S[KMAX];
  normalise(K, G, Gn);
  double best = INFINITY;
  for (int k = 0; k < K; ++k) alpha[k] = (k == 0) ? 1.0 : 0.0;
  for (uint32_t mask = 1; mask < (1u << K); ++mask) {
    int s = 0;
    for (int k = 0; k < K; ++k)
      if (mask & (1u << k)) S[s++] = k;
    if (!affine_min_norm(K, Gn, S, s, mu)) continue;
    int ok = 1;
    for (int i = 0; i < s; ++i)
      if (mu[i] < -1e-12) ok = 0;
    if (!ok) continue;
    double sum = 0.0;
    for (int k = 0; k < K; ++k) w[k] = 0.0;
    for (int i = 0; i < s; ++i) {
      w[S[i]] = mu[i] > 0.0 ? mu[i] : 0.0;
      sum += w[S[i]];
    }
    for (int k = 0; k < K; ++k) w[k] /= sum;
    double obj = quad_form(K, Gn, w);
    if (obj < best) {
      best = obj;
      memcpy(alpha, w, sizeof(double) * K);
    }
  }
}

/*
 * Frank-Wolfe replay (the iteration the GPU solver runs before its exact
 * completion; the paper names no solver).  On the normalised Gram Gn:
 *   init: the best pair.  For every i < j the K=2 closed form on (g_i, g_j)
 *     and its value; the pair of least value wins, ties to the first pair in
 *     (i, j) lexicographic order.  K = 1 gives alpha = (1).
 *   iteration: v = Gn alpha, a = alpha^T v, t = argmin_k v_k (lowest index
 *     on ties); stop when a - v_t <= tol (the duality gap); else step to
 *     (1 - gamma) alpha + gamma e_t with the exact line search
 *     gamma = clamp((a - v_t) / (a - 2 v_t + Gn_tt), 0, 1).
 * Returns the number of completed steps.
 */
int bko_mgda_fw(int32_t K, const double* G, int32_t max_iter, double tol,
                double* alpha) {
  double Gn[KMAX * KMAX], v[KMAX];
  for (int k = 0; k < K; ++k) alpha[k] = 0.0;
  if (K == 1) {
    alpha[0] = 1.0;
    return 0;
  }
  normalise(K, G, Gn);
  double best = INFINITY, bg = 0.5;
  int bi = 0, bj = 1;
  for (int i = 0; i < K; ++i)
    for (int j = i + 1; j < K; ++j) {
      double gii = Gn[i * K + i], gjj = Gn[j * K + j], gij = Gn[i * K + j];
      double den = gii + gjj - 2.0 * gij;
      double gam = 0.5;
      if (den > 0.0) {
        gam = (gjj - gij) / den;
        if (gam < 0.0) gam = 0.0;
        if (gam > 1.0) gam = 1.0;
      }
      double val = gam * gam * gii + 2.0 * gam * (1.0 - gam) * gij +
                   (1.0 - gam) * (1.0 - gam) * gjj;
      if (val < best) {
        best = val;
        bi = i;
        bj = j;
        bg = gam;
      }
    }
  alpha[bi] = bg;
  alpha[bj] = 1.0 - bg;

  int it = 0;
  for (; it < max_iter; ++it) {
    double a = 0.0;
    for (int k = 0; k < K; ++k) {
      double t = 0.0;
      for (int j = 0; j < K; ++j) t += Gn[k * K + j] * alpha[j];
      v[k] = t;
    }
    for (int k = 0; k < K; ++k) a += alpha[k] * v[k];
    int t = 0;
    for (int k = 1; k < K; ++k)
      if (v[k] < v[t]) t = k;
    double gap = a - v[t];
    if (gap <= tol) break;
    double den = a - 2.0 * v[t] + Gn[t * K + t];
    if (!(den > 0.0)) break;
    double gam = gap / den;
    if (gam > 1.0) gam = 1.0;
    for (int k = 0; k < K; ++k) alpha[k] *= (1.0 - gam);
    alpha[t] += gam;
  }
  return it;
}

/* ------------------------------------------------------------------------ */
/* PCGrad (Eq. 5; bucket form Eq. 8; the PCGrad branch of Algorithm 1).      */
/* ------------------------------------------------------------------------ */

/* SplitMix64 output function (G. Steele, D. Lea, C. Flood, "Fast splittable
 * pseudorandom number generators", OOPSLA 2014; the variant-13 mixing
 * constants published with it). */
static uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}
#define GOLDEN_GAMMA 0x9E3779B97F4A7C15ull

/*
 * The "random order" in which task t visits the other tasks (Algorithm 1,
 * PCGrad branch).  Counter-based: key = mix64 folded over (seed, step,
 * bucket, t) as k1 = mix64(seed + (step+1) G), k2 = mix64(k1 + (bucket+1) G),
 * k3 = mix64(k2 + (t+1) G) with G the golden-ratio gamma; draw i is
 * r_i = mix64(k3 + (i+1) G).  The list [0..K-1] without t, in ascending
 * order, is shuffled by Fisher-Yates from its last slot down: for
 * i = m-1 .. 1 (m = K-1) swap slot i with slot r_{m-1-i} mod (i+1).
 */
void bko_pcgrad_order(uint64_t seed, uint64_t step, int64_t bucket, int32_t K,
                      int32_t t, int32_t* order) {
  uint64_t k1 = mix64(seed + (step + 1) * GOLDEN_GAMMA);
  uint64_t k2 = mix64(k1 + ((uint64_t)bucket + 1) * GOLDEN_GAMMA);
  uint64_t k3 = mix64(k2 + ((uint64_t)t + 1) * GOLDEN_GAMMA);
  int m = 0;
  for (int k = 0; k < K; ++k)
    if (k != t) order[m++] = k;
  for (int i = m - 1, draw = 0; i >= 1; --i, ++draw) {
    uint64_t r = mix64(k3 + ((uint64_t)draw + 1) * GOLDEN_GAMMA);
    int j = (int)(r % (uint64_t)(i + 1));
    int tmp = order[i];
    order[i] = order[j];
    order[j] = tmp;
  }
}

/*
 * PCGrad on the Gram matrix.  Each running d_t = sum_m C[t][m] g_m starts as
 * g_t; for every other task j in t's order, if <d_t, g_j> < 0 it becomes
 * d_t - <d_t, g_j> / ||g_j||^2 g_j (projection onto the normal plane of the
 * ORIGINAL g_j).  <d_t, g_j> = sum_m C[t][m] G[m][j], so only G is needed.
 * A task with ||g_j|| = 0 is never projected on.  The result is
 * d = sum_t d_t (a sum, not a mean), so beta_j = sum_t C[t][j].
 * *near_ties counts tests with |<d_t, g_j>| <= 1e-6 ||d_t|| ||g_j||, where a
 * rounding difference can flip the branch.
 */
void bko_pcgrad(int32_t K, const double* G, uint64_t seed, uint64_t step,
                int64_t bucket, double* beta, int32_t* near_ties) {
  double Gn[KMAX * KMAX], C[KMAX * KMAX];
  int32_t order[KMAX];
  int32_t ties = 0;
  normalise(K, G, Gn);
  for (int i = 0; i < K * K; ++i) C[i] = 0.0;
  for (int t = 0; t < K; ++t) C[t * K + t] = 1.0;
  for (int t = 0; t < K; ++t) {
    bko_pcgrad_order(seed, step, bucket, K, t, order);
    for (int q = 0; q < K - 1; ++q) {
      int j = order[q];
      double p = 0.0;
      for (int m = 0; m < K; ++m) p += C[t * K + m] * Gn[m * K + j];
      double dd = quad_form(K, Gn, C + t * K);
      if (fabs(p) <= 1e-6 * sqrt(fabs(dd) * Gn[j * K + j])) ++ties;
      if (p < 0.0 && Gn[j * K + j] > 0.0) C[t * K + j] -= p / Gn[j * K + j];
    }
  }
  for (int j = 0; j < K; ++j) {
    double s = 0.0;
    for (int t = 0; t < K; ++t) s += C[t * K + j];
    beta[j] = s;
  }
  if (near_ties) *near_ties = ties;
}

/*
 * Every result PCGrad can give when each near-tie test may go either way.
 * The conflict test <d_t, g_j> < 0 of Eq. 5 / Algorithm 1 is discontinuous:
 * where |<d_t, g_j>| <= 1e-6 ||d_t|| ||g_j|| (the near-tie bound of
 * bko_pcgrad) a rounding difference in the Gram can flip it, and both
 * "project" and "keep" are correct outcomes.  Row t of C (the coefficients of
 * d_t) depends on no other row, so the alternatives are enumerated per task:
 * a depth-first walk of t's order that follows both branches at every near
 * tie (the projection branch only when ||g_j|| > 0), collecting the distinct
 * final rows.  beta = sum_t row_t, so the results are every sum of one
 * alternative row per task, enumerated with task 0 varying slowest.
 * Returns the number of results written to betas (n x K, row-major), or -1
 * when there are more than cap.  With no near tie the single result is
 * bko_pcgrad's.
 */
#define PCG_ROWS_MAX 64
static int pcg_rows(int K, const double* Gn, const int32_t* order, int q,
                    double* row, double* rows, int n, int cap) {
  for (; q < K - 1; ++q) {
    int j = order[q];
    double p = 0.0;
    for (int m = 0; m < K; ++m) p += row[m] * Gn[m * K + j];
    double dd = quad_form(K, Gn, row);
    int tie = fabs(p) <= 1e-6 * sqrt(fabs(dd) * Gn[j * K + j]);
    int can = Gn[j * K + j] > 0.0;
    if (tie && can) {
      double alt[KMAX];
      memcpy(alt, row, sizeof(double) * K);
      alt[j] -= p / Gn[j * K + j];
      n = pcg_rows(K, Gn, order, q + 1, alt, rows, n, cap);
      if (n < 0) return -1;
      /* the other branch continues below without the projection */
    } else if (p < 0.0 && can) {
      row[j] -= p / Gn[j * K + j];
    }
  }
  for (int i = 0; i < n; ++i) {
    int same = 1;
    for (int m = 0; m < K; ++m)
      if (rows[i * K + m] != row[m]) same = 0;
    if (same) return n;
  }
  if (n >= cap) return -1;
  memcpy(rows + n * K, row, sizeof(double) * K);
  return n + 1;
}

int32_t bko_pcgrad_alternatives(int32_t K, const double* G, uint64_t seed,
                                uint64_t step, int64_t bucket, int32_t cap,
                                double* betas) {
  double Gn[KMAX * KMAX];
  static const int rows_cap = PCG_ROWS_MAX;
  double* rows = (double*)malloc(sizeof(double) * KMAX * rows_cap * KMAX);
  int nrow[KMAX];
  int32_t order[KMAX];
  if (!rows) return -1;
  normalise(K, G, Gn);
  long total = 1;
  for (int t = 0; t < K; ++t) {
    double row[KMAX];
    for (int m = 0; m < K; ++m) row[m] = (m == t) ? 1.0 : 0.0;
    bko_pcgrad_order(seed, step, bucket, K, t, order);
    nrow[t] = pcg_rows(K, Gn, order, 0, row, rows + t * rows_cap * KMAX, 0,
                       rows_cap);
    if (nrow[t] < 0) {
      free(rows);
      return -1;
    }
    total *= nrow[t];
    if (total > cap) {
      free(rows);
      return -1;
    }
  }
  for (long r = 0; r < total; ++r) {
    int pick[KMAX];
    long rem = r;
    for (int t = K - 1; t >= 0; --t) {
      pick[t] = (int)(rem % nrow[t]);
      rem /= nrow[t];
    }
    double* out = betas + r * K;
    for (int m = 0; m < K; ++m) {
      double s = 0.0;
      for (int t = 0; t < K; ++t) s += rows[t * rows_cap * KMAX + pick[t] * K + m];
      out[m] = s;
    }
  }
  free(rows);
  return (int32_t)total;
}

/* ------------------------------------------------------------------------ */
/* CAGrad (Eq. 4; bucket form Eq. 7; the CAGrad branch of Algorithm 1).      */
/* ------------------------------------------------------------------------ */

/*
 * The primal max_d min_k <g_k, d> s.t. ||d - g0|| <= c ||g0||, g0 the mean
 * gradient, is a bilinear saddle problem over a compact convex set and the
 * simplex, so (minimax theorem) it equals
 *   min_{w in simplex} F(w),  F(w) = <g0, g_w> + rho ||g_w||,
 *   g_w = sum_k w_k g_k,  rho = c ||g0||,
 * with the maximiser d = g0 + rho g_w / ||g_w||.  On the Gram matrix:
 * <g0, g_w> = b^T w with b = G 1 / K, ||g_w||^2 = w^T G w,
 * ||g0||^2 = 1^T G 1 / K^2.  So beta = 1/K + rho w / ||g_w||.  No rescaling
 * of d is applied: the paper's definition has none.
 *
 * F is convex on the simplex.  Candidates, each a feasible point:
 *  - every vertex e_k;
 *  - for every support S with |S| >= 2 and G_SS invertible, the stationary
 *    point of F on the affine hull of S: with m = G_SS^-1 1, n = G_SS^-1 b_S,
 *    D = (1^T n)^2 - (1^T m)(n^T b_S - rho^2) > 0 and
 *    lambda = (1^T n + sqrt D) / 1^T m it is w_S = (lambda m - n) / sqrt D
 *    (from b_S + rho G_SS w_S / ||g_w|| = lambda 1, sum w_S = 1), kept when
 *    w_S >= 0;
 *  - the minimum-norm point when it is 0 (then F = 0 there).
 * The candidate of least F is returned (ties: first found).  If c = 0, or
 * g0 = 0, or the chosen g_w = 0, beta = 1/K.  w_out (may be NULL) gets w.
 * Cost 2^K solves: meant for small K and few buckets.
 */
void bko_cagrad(int32_t K, const double* G, double c, double* beta,
                double* w_out) {
  double Gn[KMAX * KMAX], b[KMAX], w[KMAX], bestw[KMAX];
  double A[KMAX * KMAX], mv[KMAX], nv[KMAX];
  int S[KMAX];
  normalise(K, G, Gn);
  double g0sq = 0.0;
  for (int i = 0; i < K; ++i) {
    double t = 0.0;
    for (int j = 0; j < K; ++j) t += Gn[i * K + j];
    b[i] = t / K;
    g0sq += t;
  }
  g0sq /= (double)K * K;
  for (int k = 0; k < K; ++k) beta[k] = 1.0 / K;
  for (int k = 0; k < K; ++k) bestw[k] = 1.0 / K;
  if (!(c > 0.0) || !(g0sq > 0.0)) {
    if (w_out) memcpy(w_out, bestw, sizeof(double) * K);
    return;
  }
  double rho = c * sqrt(g0sq);
  double bestF = INFINITY;

  for (int k = 0; k < K; ++k) {
    double F = b[k] + rho * sqrt(Gn[k * K + k] > 0.0 ? Gn[k * K + k] : 0.0);
    if (F < bestF) {
      bestF = F;
      for (int i = 0; i < K; ++i) bestw[i] = (i == k) ? 1.0 : 0.0;
    }
  }
  for (uint32_t mask = 1; mask < (1u << K); ++mask) {
    int s = 0;
    for (int k = 0; k < K; ++k)
      if (mask & (1u << k)) S[s++] = k;
    if (s < 2) continue;
    for (int i = 0; i < s; ++i)
      for (int j = 0; j < s; ++j) A[i * s + j] = Gn[S[i] * K + S[j]];
    for (int i = 0; i < s; ++i) mv[i] = 1.0;
    if (!solve_dense(s, A, mv, PIV_TOL)) continue;
    for (int i = 0; i < s; ++i)
      for (int j = 0; j < s; ++j) A[i * s + j] = Gn[S[i] * K + S[j]];
    for (int i = 0; i < s; ++i) nv[i] = b[S[i]];
    if (!solve_dense(s, A, nv, PIV_TOL)) continue;
    double om = 0.0, on = 0.0, nb = 0.0;
    for (int i = 0; i < s; ++i) {
      om += mv[i];
      on += nv[i];
      nb += nv[i] * b[S[i]];
    }
    double D = on * on - om * (nb - rho * rho);
    if (!(om > 0.0) || !(D > 0.0)) continue;
    double sd = sqrt(D);
    double lam = (on + sd) / om;
    int ok = 1;
    double sum = 0.0;
    for (int k = 0; k < K; ++k) w[k] = 0.0;
    for (int i = 0; i < s; ++i) {
      double wi = (lam * mv[i] - nv[i]) / sd;
      if (wi < -1e-12) ok = 0;
      w[S[i]] = wi > 0.0 ? wi : 0.0;
      sum += w[S[i]];
    }
    if (!ok || !(sum > 0.0)) continue;
    for (int k = 0; k < K; ++k) w[k] /= sum;
    double q = quad_form(K, Gn, w);
    double F = 0.0;
    for (int k = 0; k < K; ++k) F += b[k] * w[k];
    F += rho * sqrt(q > 0.0 ? q : 0.0);
    if (F < bestF) {
      bestF = F;
      memcpy(bestw, w, sizeof(double) * K);
    }
  }
  {
    double a[KMAX];
    if (bko_mgda_wolfe(K, G, a) >= 0) {
      double q = quad_form(K, Gn, a);
      if (q <= 1e-24) {
        double F = 0.0;
        for (int k = 0; k < K; ++k) F += b[k] * a[k];
        F += rho * sqrt(q > 0.0 ? q : 0.0);
        if (F < bestF) {
          bestF = F;
          memcpy(bestw, a, sizeof(double) * K);
        }
      }
    }
  }
  double q = quad_form(K, Gn, bestw);
  if (q > 1e-24) {
    double f = rho / sqrt(q);
    for (int k = 0; k < K; ++k) beta[k] = 1.0 / K + f * bestw[k];
  }
  if (w_out) memcpy(w_out, bestw, sizeof(double) * K);
}

/* ------------------------------------------------------------------------ */
/* Combination d_b = sum_k beta_k g_k  (Algorithm 1: the resolved update of  */
/* every rule; the concatenation d = [d_(1) .. d_(B)] of Section 3.2).       */
/* ------------------------------------------------------------------------ */

void bko_combine(int32_t K, int32_t dtype, const void* const* x,
                 int64_t begin, int64_t n, const double* beta, double* d) {
  for (int64_t e = 0; e < n; ++e) {
    double s = 0.0;
    for (int32_t k = 0; k < K; ++k)
      s += beta[k] * load_elem(x[k], dtype, begin + e);
    d[e] = s;
  }
}

/* ------------------------------------------------------------------------ */
/* Conflict statistics of Figure 1 (Eq. 2, Definition A.4).                  */
/* ------------------------------------------------------------------------ */

/*
 * Pairwise cosines cos_ij = G_ij / sqrt(G_ii G_jj) (0 when either gradient is
 * zero; 1 on the diagonal of a non-zero gradient); over the K(K-1)/2 pairs
 * i < j: mean, population standard deviation (the square root of the mean
 * squared deviation from the mean), minimum; conflict = 1 when some pair has
 * a negative cosine.  cos (K*K) may be NULL.  stats = (mean, std, min).
 */
void bko_conflicts(int32_t K, const double* G, double* cos, double* stats,
                   int32_t* conflict) {
  double c[KMAX * KMAX];
  int32_t any = 0;
  double sum = 0.0, mn = 1.0;
  int np = 0;
  for (int i = 0; i < K; ++i)
    for (int j = 0; j < K; ++j) {
      double gi = G[i * K + i], gj = G[j * K + j];
      double v;
      if (i == j) v = gi > 0.0 ? 1.0 : 0.0;
      else v = (gi > 0.0 && gj > 0.0) ? G[i * K + j] / sqrt(gi * gj) : 0.0;
      c[i * K + j] = v;
      if (i < j) {
        sum += v;
        ++np;
        if (v < mn) mn = v;
        if (v < 0.0) any = 1;
      }
    }
  double mean = np ? sum / np : 0.0, dev = 0.0;
  for (int i = 0; i < K; ++i)
    for (int j = i + 1; j < K; ++j) dev += (c[i * K + j] - mean) * (c[i * K + j] - mean);
  stats[0] = mean;
  stats[1] = np ? sqrt(dev / np) : 0.0;
  stats[2] = mn;
  if (cos) memcpy(cos, c, sizeof(double) * K * K);
  *conflict = any;
}

/* ------------------------------------------------------------------------ */
/* Whole path over buckets [b0, b1): Gram -> rule -> combination.            */
/* ------------------------------------------------------------------------ */

/*
 * x[k] are the K full flat gradients (N elements each, fp32 or bf16 bits),
 * offsets[0..B] the bucket boundaries.  Outputs (rows relative to b0):
 * beta[(b - b0) * K + k] always; gram[(b - b0) * K * K ...] and
 * d[offsets[b] - offsets[b0] + e] when non-NULL; status[b - b0] when non-NULL
 * (0, or 3 when the Gram is not finite -- then beta = 1/K).
 * n_threads > 0 runs buckets on that many OpenMP threads.
 * Returns 0, or -1 on invalid arguments.
 */
int bko_resolve(int32_t K, int32_t dtype, const void* const* x,
                const int64_t* offsets, int64_t b0, int64_t b1, int32_t rule,
                const bko_params* p, double* beta, double* d, double* gram,
                int32_t* status, int32_t n_threads) {
  if (K < 1 || K > KMAX || !x || !offsets || !p || !beta || b1 < b0) return -1;
  if (dtype != BKO_F32 && dtype != BKO_BF16) return -1;
  if (rule < BKO_MGDA || rule > BKO_MEAN) return -1;
  int64_t base = offsets[b0];
#ifdef _OPENMP
  int nt = n_threads > 0 ? n_threads : 1;
#pragma omp parallel for schedule(dynamic, 1) num_threads(nt)
#endif
  for (int64_t b = b0; b < b1; ++b) {
    double G[KMAX * KMAX], bt[KMAX];
    int64_t beg = offsets[b], n = offsets[b + 1] - offsets[b];
    bko_gram(K, dtype, x, beg, n, G);
    int32_t st = BKO_OK;
    if (!all_finite(K * K, G)) {
      st = BKO_NONFINITE;
      for (int k = 0; k < K; ++k) bt[k] = 1.0 / K;
    } else if (rule == BKO_MGDA) {
      if (K == 2 && p->mgda_mode != BKO_MGDA_FW) {
        double Gn[4];
        normalise(2, G, Gn);
        bko_mgda_k2(Gn, bt);
      } else if (p->mgda_mode == BKO_MGDA_FW) {
        bko_mgda_fw(K, G, p->max_iter, p->tol, bt);
      } else if (p->mgda_mode == BKO_MGDA_ENUM) {
        bko_mgda_enum(K, G, bt);
      } else {
        bko_mgda_wolfe(K, G, bt);
      }
    } else if (rule == BKO_PCGRAD) {
      bko_pcgrad(K, G, p->seed, p->step, b, bt, NULL);
    } else if (rule == BKO_CAGRAD) {
      bko_cagrad(K, G, p->cagrad_c, bt, NULL);
    } else {
      for (int k = 0; k < K; ++k) bt[k] = 1.0 / K;
    }
    for (int k = 0; k < K; ++k) beta[(b - b0) * K + k] = bt[k];
    if (gram) memcpy(gram + (b - b0) * K * K, G, sizeof(double) * K * K);
    if (status) status[b - b0] = st;
    if (d) bko_combine(K, dtype, x, beg, n, bt, d + (beg - base));
  }
  return 0;
}

int32_t bko_max_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}
