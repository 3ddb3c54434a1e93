"""Spectral positional encoding (SPE) of the Tanner graph, Sec. 4.3: the host precompute.

At inference the SPE vectors are a fixed table (Sec. 4.3: the learned vectors stay fixed and
add no runtime work); aecct_create takes that table (`spe`, T x d_spe) and the decoder
concatenates row t to token t's embedding.  This module computes the table on the host, in
float64, from the parity-check matrix and the SPE parameters:

  Tanner graph: T = 2n - k nodes, variable j (0 <= j < n) joined to check i (node n + i) where
  H[i, j] = 1.  Laplacian L = D - A (combinatorial).  Eigenpairs (lambda_i, phi_i), ascending.
  Phi_j in R^{T x 2}: row i = [lambda_i, phi_i[j]] (the eigenvalues beside node j's entries of the
  eigenvectors).
  X_j = Phi_j W_{2->d_SPE}                          (Q_j = K_j = V_j = X_j)
  MHSA(X_j) = Concat_e softmax((X_j Wq_e)(X_j Wk_e)^T / sqrt(d_e)) (X_j Wv_e) Wo
  SPE_j = mean over the T rows of MHSA(X_j)         (the reduction W_{(2n-k)->1}: average pooling)

Readings where Sec. 4.3 leaves the choice open: the combinatorial Laplacian; multi-head
self-attention in its standard form (per-head projections Wq_e, Wk_e, Wv_e of width
d_e = d_SPE / heads, output projection Wo, no biases); average pooling as the reduction.
Eigenvectors are fixed up to sign, and within a repeated eigenvalue up to a rotation; the
canonical basis used here removes both: for each cluster of (numerically) equal eigenvalues
with projector P, the basis is Gram-Schmidt of P e_0, P e_1, ... in node order, skipping
vectors that vanish.  For a simple eigenvalue that is the eigenvector whose first
non-vanishing entry is positive.  The basis then depends only on the graph and the node
order, not on the eigensolver.

The decoder never computes this table; the GPU precompute (aecct_spe_table) and this host
version are checked against the oracle's independent restatement.
"""
from __future__ import annotations

import math

import numpy as np

CLUSTER_TOL = 1e-8    # eigenvalues closer than this x max(1, lambda_max) form one cluster
VANISH_TOL = 1e-6     # a Gram-Schmidt residual below this norm is skipped


def tanner_laplacian(H: np.ndarray) -> np.ndarray:
    """Combinatorial Laplacian D - A of the Tanner graph (variables first, then checks)."""
    m, n = H.shape
    T = n + m
    A = np.zeros((T, T))
    Hb = (H != 0).astype(np.float64)
    A[:n, n:] = Hb.T
    A[n:, :n] = Hb
    return np.diag(A.sum(1)) - A


def canonical_eigenbasis(lam: np.ndarray, U: np.ndarray):
    """Canonical orthonormal eigenbasis from any orthonormal one (columns of U, eigenvalues lam):
    sorted ascending; per cluster of equal eigenvalues, Gram-Schmidt of P e_j in node order."""
    order = np.argsort(lam, kind="stable")
    lam = np.asarray(lam, np.float64)[order]
    U = np.asarray(U, np.float64)[:, order]
    T = lam.shape[0]
    tol = CLUSTER_TOL * max(1.0, float(np.abs(lam).max()))
    out = np.zeros_like(U)
    i = 0
    while i < T:
        j = i + 1
        while j < T and lam[j] - lam[j - 1] <= tol:
            j += 1
        Uc = U[:, i:j]
        P = Uc @ Uc.T
        basis = []
        for node in range(T):
            if len(basis) == j - i:
                break
            v = P[:, node].copy()
            for b in basis:
                v -= (b @ v) * b
            nv = math.sqrt(float(v @ v))
            if nv > VANISH_TOL:
                basis.append(v / nv)
        if len(basis) != j - i:
            raise ValueError("canonical eigenbasis: a cluster's projector has too small a range")
        out[:, i:j] = np.stack(basis, 1)
        i = j
    return lam, out


def eigenpairs(H: np.ndarray):
    """Canonical eigenpairs of the Tanner-graph Laplacian (LAPACK's symmetric solver)."""
    lam, U = np.linalg.eigh(tanner_laplacian(H))
    return canonical_eigenbasis(lam, U)


def spe_from_eigenpairs(lam: np.ndarray, U: np.ndarray, p, chunk: int = 1) -> np.ndarray:
    """SPE_j for every node j (float64, [T, d_spe]).

    Row i of X_j = Phi_j W_pe is lambda_i w0 + phi_i[j] w1 (w0, w1 the rows of W_pe), so every
    projection of it is a combination of two fixed vectors: Q_j[i] = lambda_i (w0 Wq) +
    phi_i[j] (w1 Wq), and likewise K and V.  The scores Q_j[i] . K_j[i'] are then a 2 x 2
    bilinear form in (lambda_i, phi_i[j]) and (lambda_i', phi_i'[j]), and softmax(S) V_j is
    (P lambda) (w0 Wv) + (P phi[j]) (w1 Wv): the same values as the matrix products of the
    definition, with O(T^2) work per node and head instead of O(T^2 d_e)."""
    T = lam.shape[0]
    heads, d_spe = p.wq.shape[0], p.w_pe.shape[1]
    d_e = d_spe // heads
    w0, w1 = p.w_pe[0], p.w_pe[1]
    out = np.zeros((T, d_spe))
    for j0 in range(0, T, chunk):
        Uj = U[j0:j0 + chunk]                      # [nodes, T]: phi_i[j] for every eigenvector i
        L = np.broadcast_to(lam, Uj.shape)         # [nodes, T]: lambda_i
        parts = []
        for e in range(heads):
            qa, qb = w0 @ p.wq[e], w1 @ p.wq[e]
            ka, kb = w0 @ p.wk[e], w1 @ p.wk[e]
            va, vb = w0 @ p.wv[e], w1 @ p.wv[e]
            # S[j, i, i'] = (L_i qa + U_ji qb) . (L_i' ka + U_ji' kb) / sqrt(d_e)
            Sq_a = L * (qa @ ka) + Uj * (qb @ ka)  # coefficient of L_i'
            Sq_b = L * (qa @ kb) + Uj * (qb @ kb)  # coefficient of U_ji'
            S = (Sq_a[:, :, None] * L[:, None, :] + Sq_b[:, :, None] * Uj[:, None, :]) / math.sqrt(d_e)
            S -= S.max(-1, keepdims=True)
            P = np.exp(S)
            P /= P.sum(-1, keepdims=True)
            PL = np.einsum("jab,jb->ja", P, L)     # (P lambda)_i
            PU = np.einsum("jab,jb->ja", P, Uj)    # (P phi[j])_i
            # mean over the rows i of softmax(S) V_j: mean(PL) va + mean(PU) vb
            parts.append(PL.mean(1)[:, None] * va[None, :] + PU.mean(1)[:, None] * vb[None, :])
        out[j0:j0 + chunk] = np.concatenate(parts, 1) @ p.wo
    return out


def spe_table(H: np.ndarray, params) -> np.ndarray:
    """The SPE table [T, d_spe] (float32, as aecct_create takes it) for the SPE parameters
    `params` (w_pe [2, d_spe], wq, wk, wv [heads, d_spe, d_e], wo [d_spe, d_spe])."""
    lam, U = eigenpairs(H)
    return spe_from_eigenpairs(lam, U, params).astype(np.float32)
