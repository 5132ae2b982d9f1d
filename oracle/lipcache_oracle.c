/*
 * FP64 CPU oracle for the certified cache lookup of LipCache.
 *
 * TEST INFRASTRUCTURE ONLY. This file is the plain, slow, obviously correct
 * statement of what the lookup computes. Only the tests, the smoke check and
 * the benchmark's CPU-baseline / reference arm may call it; the product
 * library never links it, and it shares no code, header or constant with the
 * CUDA path.
 *
 * Every quantity is computed from its definition in the paper, in double
 * precision, from FP32 inputs promoted exactly:
 *   - sigma_max(W): the largest singular value of the head (Sec. 4.1,
 *     Eqs. 17-19), by a one-sided (Hestenes) Jacobi SVD.
 *   - certification of a candidate row (Sec. 3.3, Algorithm 1; Eqs. 5-6,
 *     20-21; Remark 4.2, Eq. 29): all C logits, the GuardNet label, the
 *     margin, the radius, and the skip rules.
 *   - the online lookup (Sec. 3.4, Eqs. 13-15, Algorithm 2): distances by
 *     direct differences to every cached key, the hit set with the strict
 *     inequality, and the nearest hit (lowest cache index on exact ties).
 *
 * Build: gcc -std=c11 -O2 -ffp-contract=off -fopenmp -shared -fPIC.
 * -ffp-contract=off keeps every multiply and add separately rounded, so the
 * results are the same on x86-64 and AArch64.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

int orc_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}

/* ------------------------------------------------------------------------
 * Singular values of W (C x d, row-major FP32) by one-sided Jacobi.
 *
 * The n = min(C, d) vectors that are orthogonalised are the rows of W when
 * C <= d (singular values of W^T equal those of W) and the columns of W
 * otherwise. Each rotation zeroes the inner product of one pair of vectors;
 * when every pair is orthogonal to relative precision tol, the vector norms
 * are the singular values. Returns the number of sweeps used, or -1 if
 * max_sweeps was reached first. sv receives the n values in descending order.
 * ------------------------------------------------------------------------ */
static int cmp_desc(const void* a, const void* b) {
  double x = *(const double*)a, y = *(const double*)b;
  return (x < y) - (x > y);
}

int orc_singular_values(const float* W, int C, int d, double* sv, int max_sweeps) {
  const int rows_as_vectors = (C <= d);
  const int n = rows_as_vectors ? C : d; /* number of vectors */
  const int m = rows_as_vectors ? d : C; /* length of each vector */
  double* A = (double*)malloc(sizeof(double) * (size_t)n * (size_t)m);
  if (!A) return -2;
  for (int v = 0; v < n; ++v)
    for (int k = 0; k < m; ++k)
      A[(size_t)v * m + k] = rows_as_vectors ? (double)W[(size_t)v * d + k] : (double)W[(size_t)k * d + v];

  const double tol = 1e-15;
  int sweeps = 0, converged = 0;
  while (sweeps < max_sweeps) {
    int rotated = 0;
    for (int p = 0; p < n - 1; ++p) {
      for (int q = p + 1; q < n; ++q) {
        double* ap = A + (size_t)p * m;
        double* aq = A + (size_t)q * m;
        double alpha = 0.0, beta = 0.0, gamma = 0.0;
        for (int k = 0; k < m; ++k) {
          alpha += ap[k] * ap[k];
          beta += aq[k] * aq[k];
          gamma += ap[k] * aq[k];
        }
        if (gamma == 0.0 || fabs(gamma) <= tol * sqrt(alpha * beta)) continue;
        rotated = 1;
        double zeta = (beta - alpha) / (2.0 * gamma);
        double t;
        if (fabs(zeta) > 1e150) {
          t = 1.0 / (2.0 * zeta);
        } else {
          double sgn = (zeta >= 0.0) ? 1.0 : -1.0;
          t = sgn / (fabs(zeta) + sqrt(1.0 + zeta * zeta));
        }
        double c = 1.0 / sqrt(1.0 + t * t);
        double s = c * t;
        for (int k = 0; k < m; ++k) {
          double x = ap[k], y = aq[k];
          ap[k] = c * x - s * y;
          aq[k] = s * x + c * y;
        }
      }
    }
    ++sweeps;
    if (!rotated) {
      converged = 1;
      break;
    }
  }
  for (int v = 0; v < n; ++v) {
    double s2 = 0.0;
    for (int k = 0; k < m; ++k) s2 += A[(size_t)v * m + k] * A[(size_t)v * m + k];
    sv[v] = sqrt(s2);
  }
  qsort(sv, (size_t)n, sizeof(double), cmp_desc);
  free(A);
  return converged ? sweeps : -1;
}

/* sigma_max(W), the Lipschitz constant of the affine head (Eqs. 17-18; the
 * bias cancels in logit differences). Returns a negative value if the SVD
 * did not converge. */
double orc_sigma_max(const float* W, int C, int d) {
  int n = C < d ? C : d;
  double* sv = (double*)malloc(sizeof(double) * (size_t)n);
  if (!sv) return -2.0;
  int rc = orc_singular_values(W, C, d, sv, 100);
  double s = (rc < 0) ? -1.0 : sv[0];
  free(sv);
  return s;
}

/* Logits s(z) = W z + b of the affine head (Eq. 5), in FP64. */
void orc_logits(const float* W, const float* b, int C, int d, const float* z, double* s) {
  for (int c = 0; c < C; ++c) {
    double acc = 0.0;
    for (int j = 0; j < d; ++j) acc += (double)W[(size_t)c * d + j] * (double)z[j];
    s[c] = acc + (double)b[c];
  }
}

/* ------------------------------------------------------------------------
 * Certification of candidate rows (Algorithm 1, loop body).
 *
 *   y^G   = argmax_c s_c(z)                      (Eq. 6; lowest class on ties)
 *   m     = s_{y^G} - max_{j != y^G} s_j         (Eq. 20)
 *   r     = m / (sigma_max(W) * sqrt(2))         (Eq. 21, radius_mode 0)
 *   r*    = min_{j != y^G, ||W_y - W_j|| > 0} (s_y - s_j) / ||W_y - W_j||
 *                                                 (Remark 4.2, Eq. 29, mode 1;
 *                                                  +inf if every j is skipped)
 *   r    <- scale * r                            (radius tightening, Sec. 5.6)
 *   payload = caller's label if given, else the proxy label y^G (Sec. 3.3)
 *   skip if consistency is required and payload != y^G, else skip if r <= 0.
 * A row with a NaN or infinite feature has no defined margin (Eq. 20) nor
 * terms of Eq. 29: r = NaN, so it is skipped in either radius mode.
 * ------------------------------------------------------------------------ */
void orc_certify(const float* W, const float* b, int C, int d, double sigma, int radius_mode, double scale,
                 const float* H, int64_t n, const int32_t* payload, int require_consistency, int32_t* yG_out,
                 int32_t* label_out, double* margin_out, double* radius_out, int32_t* accept_out) {
  const double denom = sigma * sqrt(2.0);
#pragma omp parallel
  {
    double* s = (double*)malloc(sizeof(double) * (size_t)C);
#pragma omp for schedule(static)
    for (int64_t i = 0; i < n; ++i) {
      const float* z = H + (size_t)i * d;
      orc_logits(W, b, C, d, z, s);
      int y = 0;
      for (int c = 1; c < C; ++c)
        if (s[c] > s[y]) y = c;
      double runner = -INFINITY;
      for (int c = 0; c < C; ++c)
        if (c != y && s[c] > runner) runner = s[c];
      double m = s[y] - runner;
      double r;
      if (radius_mode == 0) {
        r = m / denom;
      } else {
        r = INFINITY;
        for (int j = 0; j < C; ++j) {
          if (j == y) continue;
          double nrm2 = 0.0;
          for (int k = 0; k < d; ++k) {
            double dw = (double)W[(size_t)y * d + k] - (double)W[(size_t)j * d + k];
            nrm2 += dw * dw;
          }
          if (nrm2 == 0.0) continue;
          double rij = (s[y] - s[j]) / sqrt(nrm2);
          if (rij < r) r = rij;
        }
      }
      int finite = 1;
      for (int k = 0; k < d; ++k)
        if (!isfinite(z[k])) finite = 0;
      if (!finite) r = NAN;
      r *= scale;
      int32_t label = payload ? payload[i] : (int32_t)y;
      int accept;
      if (require_consistency && label != y)
        accept = 0;
      else if (!(r > 0.0))
        accept = 0;
      else
        accept = 1;
      yG_out[i] = y;
      label_out[i] = label;
      margin_out[i] = m;
      radius_out[i] = r;
      accept_out[i] = accept;
    }
    free(s);
  }
}

/* Distance ||q - k||_2 by direct differences, in FP64. */
static double dist_fp64(const float* q, const float* k, int d) {
  double s = 0.0;
  for (int j = 0; j < d; ++j) {
    double t = (double)q[j] - (double)k[j];
    s += t * t;
  }
  return sqrt(s);
}

/* ------------------------------------------------------------------------
 * Online lookup (Algorithm 2, Eqs. 13-15), brute force over all N entries.
 *
 *   H(q) = { i : ||q - z_i|| < r_i }        (strict, Eq. 13)
 *   i*   = argmin_{i in H(q)} ||q - z_i||   (Eq. 14; lowest index on ties)
 *   out  = (i*, payload_{i*}, D_{i*}) on a hit, (-1, -1, +inf) on a miss
 *          (a miss means: fall back to MainNet, Eq. 15)
 *
 * Diagnostics (each output pointer may be NULL):
 *   n_hits[q]         = |H(q)|
 *   decision_band[q]  = 1 if some entry has |D - r_i| <= band_rel * r_i
 *                       (finite r_i only)
 *   selection_band[q] = 1 if |H(q)| >= 2 and the two smallest hit distances
 *                       D1 <= D2 satisfy D2 - D1 <= band_rel * D2
 * ------------------------------------------------------------------------ */
void orc_probe(const float* keys, const double* radius, const int32_t* labels, int64_t N, int d, const float* Q,
               int64_t B, int64_t* out_idx, int32_t* out_label, double* out_dist, int32_t* n_hits,
               int32_t* decision_band, int32_t* selection_band, double band_rel) {
#pragma omp parallel for schedule(dynamic, 1)
  for (int64_t qi = 0; qi < B; ++qi) {
    const float* q = Q + (size_t)qi * d;
    int64_t best = -1;
    double best_d = INFINITY, d1 = INFINITY, d2 = INFINITY;
    int32_t nh = 0, band = 0;
    for (int64_t i = 0; i < N; ++i) {
      double D = dist_fp64(q, keys + (size_t)i * d, d);
      double r = radius[i];
      if (isfinite(r) && fabs(D - r) <= band_rel * r) band = 1;
      if (D < r) {
        ++nh;
        if (D < best_d) {
          best_d = D;
          best = i;
        }
        if (D < d1) {
          d2 = d1;
          d1 = D;
        } else if (D < d2) {
          d2 = D;
        }
      }
    }
    out_idx[qi] = best;
    out_label[qi] = best >= 0 ? labels[best] : -1;
    out_dist[qi] = best >= 0 ? best_d : INFINITY;
    if (n_hits) n_hits[qi] = nh;
    if (decision_band) decision_band[qi] = band;
    if (selection_band) selection_band[qi] = (nh >= 2 && (d2 - d1) <= band_rel * d2) ? 1 : 0;
  }
}

/* D for given (query, key) pairs: out[p] = ||Q[qi[p]] - K[ki[p]]||_2. */
void orc_pair_dist(const float* Q, const float* K, int d, const int64_t* qi, const int64_t* ki, int64_t npairs,
                   double* out) {
#pragma omp parallel for schedule(static)
  for (int64_t p = 0; p < npairs; ++p) out[p] = dist_fp64(Q + (size_t)qi[p] * d, K + (size_t)ki[p] * d, d);
}
