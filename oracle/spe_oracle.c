/*
 * Spectral positional encoding of the Tanner graph -- CPU ORACLE.  TEST INFRASTRUCTURE ONLY.
 *
 * The plain, slow reference for the SPE table (Sec. 4.3 of "Accelerating Error Correction Code
 * Transformers"), in double precision.  Only the tests load it.  It shares no code with the
 * CUDA library or with the package's host precompute (paper_2410_05911_gb300/spe.py, which uses
 * LAPACK and an algebraic shortcut); this file uses its own eigensolver (cyclic Jacobi
 * rotations) and the definition written out step by step:
 *
 *   Tanner graph: nodes 0..n-1 are the variables, n..n+m-1 the checks; variable j and check i
 *   are joined where H[i][j] = 1.  L = D - A.
 *   Eigenpairs (lambda_i, phi_i) of L, ascending, in the canonical basis: for every cluster of
 *   equal eigenvalues (consecutive gaps <= cluster_tol), Gram-Schmidt of P e_0, P e_1, ... (P the
 *   cluster's projector), skipping residuals of norm <= vanish_tol.
 *   For each node j: Phi_j [T][2], row i = (lambda_i, phi_i[j]); X = Phi_j W_pe [T][d_spe];
 *   per head e: Q = X Wq_e, K = X Wk_e, V = X Wv_e [T][d_e];
 *   A_e = softmax_rows(Q K^T / sqrt(d_e)) V; Y = [A_0 .. A_{h-1}] Wo [T][d_spe];
 *   SPE_j = (1/T) sum over the rows of Y.
 *
 * Pins (tests/test_spe.py): L v = lambda v and orthonormality, the trace and the zero
 * eigenvalue of a connected graph, LAPACK's eigenvalues on the same matrix, the invariance of
 * the canonical basis under rotations within a cluster, closed forms of the SPE with uniform
 * attention and with the eigenvector column switched off.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* Combinatorial Laplacian of the Tanner graph of H (m x n, row-major 0/1), T = n + m. */
void spe_oracle_laplacian(const uint8_t *H, int n, int m, double *L) {
  const int T = n + m;
  memset(L, 0, sizeof(double) * (size_t)T * T);
  for (int i = 0; i < m; ++i)
    for (int j = 0; j < n; ++j)
      if (H[(size_t)i * n + j]) {
        const int c = n + i;
        L[(size_t)j * T + c] -= 1.0;
        L[(size_t)c * T + j] -= 1.0;
        L[(size_t)j * T + j] += 1.0;
        L[(size_t)c * T + c] += 1.0;
      }
}

/* Cyclic Jacobi eigenvalue algorithm for a symmetric T x T matrix S (overwritten).  On return
 * lam[i] holds the eigenvalues (unsorted) and column i of V (row-major, V[r*T + i]) the unit
 * eigenvector of lam[i].  Sweeps over all pairs (p, q) rotate away S[p][q]; stops when the
 * off-diagonal sum of squares is below 1e-30 times the squared Frobenius norm, or after 100
 * sweeps.  Returns the number of sweeps. */
int spe_oracle_jacobi(double *S, int T, double *lam, double *V) {
  double fro = 0.0;
  for (size_t i = 0; i < (size_t)T * T; ++i) fro += S[i] * S[i];
  for (int r = 0; r < T; ++r)
    for (int c = 0; c < T; ++c) V[(size_t)r * T + c] = (r == c) ? 1.0 : 0.0;
  int sweep = 0;
  for (; sweep < 100; ++sweep) {
    double off = 0.0;
    for (int p = 0; p < T; ++p)
      for (int q = p + 1; q < T; ++q) off += 2.0 * S[(size_t)p * T + q] * S[(size_t)p * T + q];
    if (off <= 1e-30 * fro) break;
    for (int p = 0; p < T; ++p)
      for (int q = p + 1; q < T; ++q) {
        const double apq = S[(size_t)p * T + q];
        if (apq == 0.0) continue;
        const double app = S[(size_t)p * T + p], aqq = S[(size_t)q * T + q];
        /* the rotation angle that zeroes S[p][q]: t = tan(theta), the smaller root of
           t^2 + 2 tau t - 1 = 0, tau = (aqq - app) / (2 apq) */
        const double tau = (aqq - app) / (2.0 * apq);
        const double t = (tau >= 0.0 ? 1.0 : -1.0) / (fabs(tau) + sqrt(1.0 + tau * tau));
        const double c = 1.0 / sqrt(1.0 + t * t), s = t * c;
        for (int k = 0; k < T; ++k) {  /* columns p and q of S */
          const double skp = S[(size_t)k * T + p], skq = S[(size_t)k * T + q];
          S[(size_t)k * T + p] = c * skp - s * skq;
          S[(size_t)k * T + q] = s * skp + c * skq;
        }
        for (int k = 0; k < T; ++k) {  /* rows p and q of S */
          const double spk = S[(size_t)p * T + k], sqk = S[(size_t)q * T + k];
          S[(size_t)p * T + k] = c * spk - s * sqk;
          S[(size_t)q * T + k] = s * spk + c * sqk;
        }
        for (int k = 0; k < T; ++k) {  /* accumulate the eigenvectors */
          const double vkp = V[(size_t)k * T + p], vkq = V[(size_t)k * T + q];
          V[(size_t)k * T + p] = c * vkp - s * vkq;
          V[(size_t)k * T + q] = s * vkp + c * vkq;
        }
      }
  }
  for (int i = 0; i < T; ++i) lam[i] = S[(size_t)i * T + i];
  return sweep;
}

/* Sort eigenpairs ascending (stable selection of the smallest remaining), then replace each
 * cluster's basis by the canonical one.  lam [T], V [T][T] (column i = eigenvector i) in place.
 * Returns 0, or -1 when a cluster's projector yields fewer vectors than its size. */
int spe_oracle_canonical(double *lam, double *V, int T, double cluster_tol, double vanish_tol) {
  double *tmp = (double *)malloc(sizeof(double) * (size_t)T);
  for (int i = 0; i < T; ++i) {
    int best = i;
    for (int j = i + 1; j < T; ++j)
      if (lam[j] < lam[best]) best = j;
    if (best != i) {
      /* move pair `best` to position i, shifting i..best-1 up by one (keeps the order stable) */
      const double lb = lam[best];
      for (int r = 0; r < T; ++r) tmp[r] = V[(size_t)r * T + best];
      for (int j = best; j > i; --j) {
        lam[j] = lam[j - 1];
        for (int r = 0; r < T; ++r) V[(size_t)r * T + j] = V[(size_t)r * T + j - 1];
      }
      lam[i] = lb;
      for (int r = 0; r < T; ++r) V[(size_t)r * T + i] = tmp[r];
    }
  }
  double amax = 1.0;
  for (int i = 0; i < T; ++i)
    if (fabs(lam[i]) > amax) amax = fabs(lam[i]);
  const double tol = cluster_tol * amax;
  double *P = (double *)malloc(sizeof(double) * (size_t)T * T);
  double *B = (double *)malloc(sizeof(double) * (size_t)T * T); /* chosen vectors, one per row */
  int rc = 0;
  int i = 0;
  while (i < T) {
    int j = i + 1;
    while (j < T && lam[j] - lam[j - 1] <= tol) ++j;
    const int r = j - i;
    /* P = sum over the cluster's columns of v v^T */
    for (int a = 0; a < T; ++a)
      for (int b = 0; b < T; ++b) {
        double s = 0.0;
        for (int c = i; c < j; ++c) s += V[(size_t)a * T + c] * V[(size_t)b * T + c];
        P[(size_t)a * T + b] = s;
      }
    int got = 0;
    for (int node = 0; node < T && got < r; ++node) {
      for (int a = 0; a < T; ++a) tmp[a] = P[(size_t)a * T + node]; /* P e_node */
      for (int g = 0; g < got; ++g) {                               /* minus its projections */
        double dot = 0.0;
        for (int a = 0; a < T; ++a) dot += B[(size_t)g * T + a] * tmp[a];
        for (int a = 0; a < T; ++a) tmp[a] -= dot * B[(size_t)g * T + a];
      }
      double nv = 0.0;
      for (int a = 0; a < T; ++a) nv += tmp[a] * tmp[a];
      nv = sqrt(nv);
      if (nv > vanish_tol) {
        for (int a = 0; a < T; ++a) B[(size_t)got * T + a] = tmp[a] / nv;
        ++got;
      }
    }
    if (got != r) rc = -1;
    for (int g = 0; g < got; ++g)
      for (int a = 0; a < T; ++a) V[(size_t)a * T + i + g] = B[(size_t)g * T + a];
    i = j;
  }
  free(tmp);
  free(P);
  free(B);
  return rc;
}

/* SPE_j of the nodes listed in `nodes` (count nn), from canonical eigenpairs lam [T], V [T][T]
 * and the parameters W_pe [2][d_spe], Wq, Wk, Wv [heads][d_spe][d_e], Wo [d_spe][d_spe]
 * (all row-major).  out [nn][d_spe]. */
void spe_oracle_mhsa(const double *lam, const double *V, int T, const int *nodes, int nn, int d_spe, int heads,
                     const double *W_pe, const double *Wq, const double *Wk, const double *Wv, const double *Wo,
                     double *out) {
  const int d_e = d_spe / heads;
  double *X = (double *)malloc(sizeof(double) * (size_t)T * d_spe);
  double *Q = (double *)malloc(sizeof(double) * (size_t)T * d_e);
  double *K = (double *)malloc(sizeof(double) * (size_t)T * d_e);
  double *Vh = (double *)malloc(sizeof(double) * (size_t)T * d_e);
  double *Acat = (double *)malloc(sizeof(double) * (size_t)T * d_spe);
  double *srow = (double *)malloc(sizeof(double) * (size_t)T);
  const double scale = 1.0 / sqrt((double)d_e);
  for (int jj = 0; jj < nn; ++jj) {
    const int j = nodes[jj];
    /* X = Phi_j W_pe, Phi_j row i = (lambda_i, phi_i[j]) */
    for (int i = 0; i < T; ++i)
      for (int c = 0; c < d_spe; ++c)
        X[(size_t)i * d_spe + c] = lam[i] * W_pe[c] + V[(size_t)j * T + i] * W_pe[d_spe + c];
    for (int e = 0; e < heads; ++e) {
      const double *wq = Wq + (size_t)e * d_spe * d_e, *wk = Wk + (size_t)e * d_spe * d_e,
                   *wv = Wv + (size_t)e * d_spe * d_e;
      for (int i = 0; i < T; ++i)
        for (int c = 0; c < d_e; ++c) {
          double sq = 0.0, sk = 0.0, sv = 0.0;
          for (int a = 0; a < d_spe; ++a) {
            const double x = X[(size_t)i * d_spe + a];
            sq += x * wq[(size_t)a * d_e + c];
            sk += x * wk[(size_t)a * d_e + c];
            sv += x * wv[(size_t)a * d_e + c];
          }
          Q[(size_t)i * d_e + c] = sq, K[(size_t)i * d_e + c] = sk, Vh[(size_t)i * d_e + c] = sv;
        }
      for (int i = 0; i < T; ++i) {
        double mx = -INFINITY;
        for (int u = 0; u < T; ++u) {
          double s = 0.0;
          for (int c = 0; c < d_e; ++c) s += Q[(size_t)i * d_e + c] * K[(size_t)u * d_e + c];
          srow[u] = s * scale;
          if (srow[u] > mx) mx = srow[u];
        }
        double l = 0.0;
        for (int u = 0; u < T; ++u) {
          srow[u] = exp(srow[u] - mx);
          l += srow[u];
        }
        for (int c = 0; c < d_e; ++c) {
          double s = 0.0;
          for (int u = 0; u < T; ++u) s += srow[u] * Vh[(size_t)u * d_e + c];
          Acat[(size_t)i * d_spe + e * d_e + c] = s / l;
        }
      }
    }
    for (int c = 0; c < d_spe; ++c) {
      double s = 0.0;
      for (int i = 0; i < T; ++i) {
        double y = 0.0;
        for (int a = 0; a < d_spe; ++a) y += Acat[(size_t)i * d_spe + a] * Wo[(size_t)a * d_spe + c];
        s += y;
      }
      out[(size_t)jj * d_spe + c] = s / (double)T;
    }
  }
  free(X);
  free(Q);
  free(K);
  free(Vh);
  free(Acat);
  free(srow);
}

/* The whole precompute: Laplacian, Jacobi, canonical basis, SPE of the listed nodes.
 * lam [T] and V [T][T] receive the canonical eigenpairs.  Returns the Jacobi sweeps, or -1. */
int spe_oracle_table(const uint8_t *H, int n, int m, int d_spe, int heads, const double *W_pe, const double *Wq,
                     const double *Wk, const double *Wv, const double *Wo, double cluster_tol, double vanish_tol,
                     const int *nodes, int nn, double *lam, double *V, double *out) {
  const int T = n + m;
  double *S = (double *)malloc(sizeof(double) * (size_t)T * T);
  spe_oracle_laplacian(H, n, m, S);
  const int sweeps = spe_oracle_jacobi(S, T, lam, V);
  free(S);
  if (spe_oracle_canonical(lam, V, T, cluster_tol, vanish_tol) != 0) return -1;
  spe_oracle_mhsa(lam, V, T, nodes, nn, d_spe, heads, W_pe, Wq, Wk, Wv, Wo, out);
  return sweeps;
}
