// spe.cu -- the spectral positional encoding of Sec. 4.3 computed on the GPU (aecct_spe_table), in
// double precision:
//
//   jacobi_kernel     eigenpairs of the Tanner-graph Laplacian L = D - A by the parallel (two-sided)
//                     Jacobi method: every step rotates n/2 disjoint index pairs (p, q) of a
//                     round-robin tournament, each rotation chosen from the current 2 x 2 block so
//                     that A[p][q] becomes 0, applied to the rows, then the columns of A and of the
//                     eigenvector matrix V; a sweep is n - 1 steps; sweeps repeat until the
//                     off-diagonal sum of squares is below 1e-30 of the Frobenius norm squared.  One
//                     cooperative launch, grid-wide barriers between the phases.
//   sort_kernel       eigenpairs in ascending order (rank by counting, ties by index).
//   canonical_kernel  per cluster of equal eigenvalues (consecutive gaps <= cluster_tol x
//                     max(1, |lambda|max)), the canonical basis: Gram-Schmidt of P e_0, P e_1, ...
//                     in node order, P = U_c U_c^T the cluster's projector, skipping residuals of
//                     norm <= vanish_tol (projections removed twice, "twice is enough").
//   mhsa_kernel       SPE_j = mean over rows of MHSA(Phi_j W_pe), Phi_j row i = (lambda_i, phi_i[j]):
//                     every projection of row i is lambda_i (w0 W) + phi_i[j] (w1 W) for the rows
//                     w0, w1 of W_pe, so each head's scores are a 2 x 2 bilinear form and
//                     softmax(S) V_j = (P lambda)(w0 Wv) + (P phi[j])(w1 Wv); two passes per query
//                     row (maximum, then the sums).
#include <cooperative_groups.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>
#include <vector>

#include "aecct_internal.h"

namespace cg = cooperative_groups;

namespace aecct {

namespace {

constexpr int kJacobiThreads = 256;
constexpr int kMaxSweeps = 100;

// index of player k at step s of the round-robin tournament on n players (player 0 stays put)
__device__ __forceinline__ int rr_player(int k, int s, int n) { return k == 0 ? 0 : ((k - 1 + s) % (n - 1)) + 1; }

__global__ void __launch_bounds__(kJacobiThreads) jacobi_kernel(double *A, double *V, int T, int n, double *cs,
                                                               double *acc, int *sweeps_out) {
  cg::grid_group grid = cg::this_grid();
  const int64_t tid = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  const int64_t nthreads = static_cast<int64_t>(gridDim.x) * blockDim.x;
  __shared__ double red[kJacobiThreads / 32];
  auto block_sum_atomic = [&](double v, double *dst) {
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
    __syncthreads();
    if (threadIdx.x == 0) {
      double s = 0.0;
      for (int w = 0; w < kJacobiThreads / 32; ++w) s += red[w];
      atomicAdd(dst, s);
    }
    __syncthreads();
  };
  // acc[0]: Frobenius norm squared; acc[1 + s]: off-diagonal sum of squares before sweep s
  {
    double f = 0.0;
    for (int64_t i = tid; i < static_cast<int64_t>(T) * T; i += nthreads) f += A[i] * A[i];
    block_sum_atomic(f, acc);
  }
  int sweep = 0;
  for (; sweep < kMaxSweeps; ++sweep) {
    grid.sync();
    double off = 0.0;
    for (int64_t i = tid; i < static_cast<int64_t>(T) * T; i += nthreads) {
      const int r = static_cast<int>(i / T), c = static_cast<int>(i % T);
      if (r != c) off += A[i] * A[i];
    }
    block_sum_atomic(off, acc + 1 + sweep);
    grid.sync();
    if (acc[1 + sweep] <= 1e-30 * acc[0]) break;
    for (int s = 0; s < n - 1; ++s) {
      // the rotations of this step (a pair with the padding player n - 1 >= T does nothing)
      for (int64_t k = tid; k < n / 2; k += nthreads) {
        int p = rr_player(static_cast<int>(k), s, n), q = rr_player(n - 1 - static_cast<int>(k), s, n);
        double c = 1.0, sn = 0.0;
        if (p < T && q < T) {
          const double apq = A[static_cast<int64_t>(p) * T + q];
          if (apq != 0.0) {
            const double app = A[static_cast<int64_t>(p) * T + p], aqq = A[static_cast<int64_t>(q) * T + q];
            const double tau = (aqq - app) / (2.0 * apq);
            const double t = (tau >= 0.0 ? 1.0 : -1.0) / (fabs(tau) + sqrt(1.0 + tau * tau));
            c = 1.0 / sqrt(1.0 + t * t);
            sn = t * c;
          }
        }
        cs[2 * k] = c;
        cs[2 * k + 1] = sn;
      }
      grid.sync();
      // rows p and q of A
      for (int64_t it = tid; it < static_cast<int64_t>(n / 2) * T; it += nthreads) {
        const int k = static_cast<int>(it / T), col = static_cast<int>(it % T);
        const int p = rr_player(k, s, n), q = rr_player(n - 1 - k, s, n);
        if (p >= T || q >= T) continue;
        const double c = cs[2 * k], sn = cs[2 * k + 1];
        const double apk = A[static_cast<int64_t>(p) * T + col], aqk = A[static_cast<int64_t>(q) * T + col];
        A[static_cast<int64_t>(p) * T + col] = c * apk - sn * aqk;
        A[static_cast<int64_t>(q) * T + col] = sn * apk + c * aqk;
      }
      grid.sync();
      // columns p and q of A and of V
      for (int64_t it = tid; it < static_cast<int64_t>(n / 2) * T; it += nthreads) {
        const int k = static_cast<int>(it / T), row = static_cast<int>(it % T);
        const int p = rr_player(k, s, n), q = rr_player(n - 1 - k, s, n);
        if (p >= T || q >= T) continue;
        const double c = cs[2 * k], sn = cs[2 * k + 1];
        const int64_t rp = static_cast<int64_t>(row) * T + p, rq = static_cast<int64_t>(row) * T + q;
        const double akp = A[rp], akq = A[rq];
        A[rp] = c * akp - sn * akq;
        A[rq] = sn * akp + c * akq;
        const double vkp = V[rp], vkq = V[rq];
        V[rp] = c * vkp - sn * vkq;
        V[rq] = sn * vkp + c * vkq;
      }
      grid.sync();
    }
  }
  if (tid == 0) *sweeps_out = sweep;
}

// ascending order: rank of eigenvalue i = #{j : lam_j < lam_i, or lam_j == lam_i and j < i}
__global__ void sort_kernel(const double *A, const double *V, int T, double *lam, double *U) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= T) return;
  const double li = A[static_cast<int64_t>(i) * T + i];
  int rank = 0;
  for (int j = 0; j < T; ++j) {
    const double lj = A[static_cast<int64_t>(j) * T + j];
    rank += (lj < li || (lj == li && j < i)) ? 1 : 0;
  }
  lam[rank] = li;
  for (int r = 0; r < T; ++r) U[static_cast<int64_t>(r) * T + rank] = V[static_cast<int64_t>(r) * T + i];
}

// block-wide sum of one double per thread (every thread gets the result)
__device__ double block_sum(double v, double *red) {
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
  __syncthreads();
  double s = 0.0;
  for (int w = 0; w < static_cast<int>(blockDim.x >> 5); ++w) s += red[w];
  __syncthreads();
  return s;
}

// one CTA per eigenvalue index i; the CTA of a cluster's first index builds its canonical basis
__global__ void canonical_kernel(const double *lam, const double *U, int T, double cluster_tol, double vanish_tol,
                                 double *Uc, double *vbuf, double *dots, int *status) {
  __shared__ double red[32];
  const int i = blockIdx.x;
  double amax = 1.0;
  for (int j = 0; j < T; ++j) amax = fmax(amax, fabs(lam[j]));
  const double tol = cluster_tol * amax;
  if (i > 0 && lam[i] - lam[i - 1] <= tol) return;  // not the first index of its cluster
  int j1 = i + 1;
  while (j1 < T && lam[j1] - lam[j1 - 1] <= tol) ++j1;
  const int r = j1 - i;
  double *v = vbuf + static_cast<int64_t>(i) * T;  // this cluster's working vector
  double *dt = dots + static_cast<int64_t>(i) * T;  // its projection coefficients (r <= T)
  int got = 0;
  for (int node = 0; node < T && got < r; ++node) {
    // v = P e_node = U_c (U_c^T e_node): column a of the cluster weighted by U[node][a]
    for (int a = threadIdx.x; a < T; a += blockDim.x) {
      double s = 0.0;
      for (int c = i; c < j1; ++c) s += U[static_cast<int64_t>(a) * T + c] * U[static_cast<int64_t>(node) * T + c];
      v[a] = s;
    }
    __syncthreads();
    // remove the projections on the vectors chosen so far, twice (one warp per coefficient)
    for (int pass = 0; pass < 2 && got > 0; ++pass) {
      const int lane = threadIdx.x & 31, nw = blockDim.x >> 5;
      for (int b = threadIdx.x >> 5; b < got; b += nw) {
        double s = 0.0;
        for (int a = lane; a < T; a += 32) s += Uc[static_cast<int64_t>(a) * T + i + b] * v[a];
        for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
        if (lane == 0) dt[b] = s;
      }
      __syncthreads();
      for (int a = threadIdx.x; a < T; a += blockDim.x) {
        double s = v[a];
        for (int b = 0; b < got; ++b) s -= dt[b] * Uc[static_cast<int64_t>(a) * T + i + b];
        v[a] = s;
      }
      __syncthreads();
    }
    double nv = 0.0;
    for (int a = threadIdx.x; a < T; a += blockDim.x) nv += v[a] * v[a];
    nv = sqrt(block_sum(nv, red));
    if (nv > vanish_tol) {
      for (int a = threadIdx.x; a < T; a += blockDim.x) Uc[static_cast<int64_t>(a) * T + i + got] = v[a] / nv;
      ++got;
    }
    __syncthreads();
  }
  if (got != r && threadIdx.x == 0) atomicOr(status, 1);
}

struct MhsaCoef {
  // per head: the score form (alpha, beta, gamma, delta) / sqrt(d_e) and the value rows va, vb
  double form[kSpeMaxHeads][4];
};

// one CTA per node j: SPE_j[c] = sum_e sum_k (mean_i PL_i va_e[k] + mean_i PU_i vb_e[k]) Wo[e d_e + k][c]
__global__ void mhsa_kernel(const double *lam, const double *U, int T, int heads, const MhsaCoef coef,
                            const double *va, const double *vb, const double *wo, int d_spe, float *spe,
                            double *spe64) {
  extern __shared__ double sh[];
  double *L = sh, *u = sh + T;
  __shared__ double red[32], mean[2 * kSpeMaxHeads];
  const int j = blockIdx.x;
  for (int a = threadIdx.x; a < T; a += blockDim.x) {
    L[a] = lam[a];
    u[a] = U[static_cast<int64_t>(j) * T + a];  // phi_a[j]
  }
  __syncthreads();
  for (int e = 0; e < heads; ++e) {
    const double al = coef.form[e][0], be = coef.form[e][1], ga = coef.form[e][2], de = coef.form[e][3];
    double spl = 0.0, spu = 0.0;
    for (int i = threadIdx.x; i < T; i += blockDim.x) {
      // s_i' = (L_i al + u_i ga) L_i' + (L_i be + u_i de) u_i'
      const double A1 = L[i] * al + u[i] * ga, B1 = L[i] * be + u[i] * de;
      double m = -INFINITY;
      for (int k = 0; k < T; ++k) m = fmax(m, A1 * L[k] + B1 * u[k]);
      double l = 0.0, pl = 0.0, pu = 0.0;
      for (int k = 0; k < T; ++k) {
        const double p = exp(A1 * L[k] + B1 * u[k] - m);
        l += p;
        pl += p * L[k];
        pu += p * u[k];
      }
      spl += pl / l;
      spu += pu / l;
    }
    spl = block_sum(spl, red);
    spu = block_sum(spu, red);
    if (threadIdx.x == 0) mean[2 * e] = spl / T, mean[2 * e + 1] = spu / T;
  }
  __syncthreads();
  const int d_e = d_spe / heads;
  for (int c = threadIdx.x; c < d_spe; c += blockDim.x) {
    double s = 0.0;
    for (int e = 0; e < heads; ++e)
      for (int k = 0; k < d_e; ++k)
        s += (mean[2 * e] * va[e * d_e + k] + mean[2 * e + 1] * vb[e * d_e + k]) * wo[(e * d_e + k) * d_spe + c];
    spe[static_cast<int64_t>(j) * d_spe + c] = static_cast<float>(s);
    if (spe64) spe64[static_cast<int64_t>(j) * d_spe + c] = s;
  }
}

}  // namespace

cudaError_t run_spe_table(const uint8_t *H, int n, int m, int d_spe, int heads, const double *w_pe, const double *wq,
                          const double *wk, const double *wv, const double *wo, double cluster_tol, double vanish_tol,
                          float *spe_host, double *lam_host, double *U_host, double *spe64_host, int *sweeps,
                          int *status_host) {
  const int T = n + m, np = T + (T & 1);
  const int d_e = d_spe / heads;
  // the Laplacian on the host (a T x T 0/1 pattern), everything after it on the device
  std::vector<double> Lh(static_cast<size_t>(T) * T, 0.0), Vh(static_cast<size_t>(T) * T, 0.0);
  for (int i = 0; i < m; ++i)
    for (int j = 0; j < n; ++j)
      if (H[static_cast<size_t>(i) * n + j]) {
        const int c = n + i;
        Lh[static_cast<size_t>(j) * T + c] -= 1.0, Lh[static_cast<size_t>(c) * T + j] -= 1.0;
        Lh[static_cast<size_t>(j) * T + j] += 1.0, Lh[static_cast<size_t>(c) * T + c] += 1.0;
      }
  for (int i = 0; i < T; ++i) Vh[static_cast<size_t>(i) * T + i] = 1.0;
  // the projections of the two rows of W_pe and the score forms per head
  MhsaCoef coef = {};
  std::vector<double> vah(static_cast<size_t>(d_spe)), vbh(static_cast<size_t>(d_spe));
  for (int e = 0; e < heads; ++e) {
    std::vector<double> qa(d_e), qb(d_e), ka(d_e), kb(d_e);
    for (int k = 0; k < d_e; ++k) {
      double s[6] = {0, 0, 0, 0, 0, 0};
      for (int a = 0; a < d_spe; ++a) {
        const size_t idx = (static_cast<size_t>(e) * d_spe + a) * d_e + k;
        s[0] += w_pe[a] * wq[idx], s[1] += w_pe[d_spe + a] * wq[idx];
        s[2] += w_pe[a] * wk[idx], s[3] += w_pe[d_spe + a] * wk[idx];
        s[4] += w_pe[a] * wv[idx], s[5] += w_pe[d_spe + a] * wv[idx];
      }
      qa[k] = s[0], qb[k] = s[1], ka[k] = s[2], kb[k] = s[3], vah[e * d_e + k] = s[4], vbh[e * d_e + k] = s[5];
    }
    double f[4] = {0, 0, 0, 0};
    for (int k = 0; k < d_e; ++k) f[0] += qa[k] * ka[k], f[1] += qa[k] * kb[k], f[2] += qb[k] * ka[k], f[3] += qb[k] * kb[k];
    const double sc = 1.0 / std::sqrt(static_cast<double>(d_e));
    for (int t = 0; t < 4; ++t) coef.form[e][t] = f[t] * sc;
  }
  double *A = nullptr, *V = nullptr, *U = nullptr, *Uc = nullptr, *lam = nullptr, *cs = nullptr, *acc = nullptr;
  double *vbuf = nullptr, *dots = nullptr, *va = nullptr, *vb = nullptr, *wod = nullptr, *spe64 = nullptr;
  float *spe = nullptr;
  int *dsweeps = nullptr, *dstatus = nullptr;
  const size_t TT = static_cast<size_t>(T) * T * sizeof(double);
  cudaError_t e = cudaSuccess;
  int dev = 0, sms = 0, per_sm = 0;
  auto ok = [&](cudaError_t x) { return (e = x) == cudaSuccess; };
  if (!ok(cudaMalloc(&A, TT)) || !ok(cudaMalloc(&V, TT)) || !ok(cudaMalloc(&U, TT)) || !ok(cudaMalloc(&Uc, TT)) ||
      !ok(cudaMalloc(&vbuf, TT)) || !ok(cudaMalloc(&dots, TT)) || !ok(cudaMalloc(&lam, sizeof(double) * T)) ||
      !ok(cudaMalloc(&cs, sizeof(double) * np)) || !ok(cudaMalloc(&acc, sizeof(double) * (kMaxSweeps + 1))) ||
      !ok(cudaMalloc(&va, sizeof(double) * d_spe)) || !ok(cudaMalloc(&vb, sizeof(double) * d_spe)) ||
      !ok(cudaMalloc(&wod, sizeof(double) * d_spe * d_spe)) || !ok(cudaMalloc(&spe, sizeof(float) * T * d_spe)) ||
      !ok(cudaMalloc(&spe64, sizeof(double) * T * d_spe)) || !ok(cudaMalloc(&dsweeps, sizeof(int))) ||
      !ok(cudaMalloc(&dstatus, sizeof(int))))
    goto done;
  if (!ok(cudaMemcpy(A, Lh.data(), TT, cudaMemcpyHostToDevice)) || !ok(cudaMemcpy(V, Vh.data(), TT, cudaMemcpyHostToDevice)) ||
      !ok(cudaMemset(acc, 0, sizeof(double) * (kMaxSweeps + 1))) || !ok(cudaMemset(dstatus, 0, sizeof(int))) ||
      !ok(cudaMemset(Uc, 0, TT)) ||
      !ok(cudaMemcpy(va, vah.data(), sizeof(double) * d_spe, cudaMemcpyHostToDevice)) ||
      !ok(cudaMemcpy(vb, vbh.data(), sizeof(double) * d_spe, cudaMemcpyHostToDevice)) ||
      !ok(cudaMemcpy(wod, wo, sizeof(double) * d_spe * d_spe, cudaMemcpyHostToDevice)))
    goto done;
  if (!ok(cudaGetDevice(&dev)) || !ok(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) ||
      !ok(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, jacobi_kernel, kJacobiThreads, 0)))
    goto done;
  {
    int Targ = T, narg = np;
    void *args[] = {&A, &V, &Targ, &narg, &cs, &acc, &dsweeps};
    const int blocks = sms * (per_sm < 2 ? per_sm : 2);
    if (!ok(cudaLaunchCooperativeKernel(reinterpret_cast<void *>(jacobi_kernel), dim3(blocks), dim3(kJacobiThreads), args,
                                        0, nullptr)))
      goto done;
  }
  sort_kernel<<<(T + 127) / 128, 128>>>(A, V, T, lam, U);
  canonical_kernel<<<T, 256>>>(lam, U, T, cluster_tol, vanish_tol, Uc, vbuf, dots, dstatus);
  mhsa_kernel<<<T, 256, 2 * sizeof(double) * T>>>(lam, Uc, T, heads, coef, va, vb, wod, d_spe, spe, spe64);
  if (!ok(cudaGetLastError()) || !ok(cudaDeviceSynchronize())) goto done;
  if (!ok(cudaMemcpy(spe_host, spe, sizeof(float) * T * d_spe, cudaMemcpyDeviceToHost)) ||
      !ok(cudaMemcpy(sweeps, dsweeps, sizeof(int), cudaMemcpyDeviceToHost)) ||
      !ok(cudaMemcpy(status_host, dstatus, sizeof(int), cudaMemcpyDeviceToHost)))
    goto done;
  if (lam_host && !ok(cudaMemcpy(lam_host, lam, sizeof(double) * T, cudaMemcpyDeviceToHost))) goto done;
  if (U_host && !ok(cudaMemcpy(U_host, Uc, TT, cudaMemcpyDeviceToHost))) goto done;
  if (spe64_host && !ok(cudaMemcpy(spe64_host, spe64, sizeof(double) * T * d_spe, cudaMemcpyDeviceToHost))) goto done;
done:
  cudaFree(A), cudaFree(V), cudaFree(U), cudaFree(Uc), cudaFree(vbuf), cudaFree(dots), cudaFree(lam), cudaFree(cs);
  cudaFree(acc), cudaFree(va), cudaFree(vb), cudaFree(wod), cudaFree(spe), cudaFree(spe64), cudaFree(dsweeps);
  cudaFree(dstatus);
  return e;
}

}  // namespace aecct
