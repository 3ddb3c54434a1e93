"""The spectral positional encoding of Sec. 4.3: the oracle (oracle/spe_oracle.c) against what
the mathematics fixes, then the package's host precompute (paper_2410_05911_gb300.spe) against
the oracle.

Pins of the oracle:
* its Jacobi eigenpairs satisfy L v = lambda v with orthonormal v; the eigenvalues sum to
  trace(L) = 2|E|; a connected Tanner graph has one zero eigenvalue, with the constant vector;
  the eigenvalues equal LAPACK's (numpy.linalg.eigvalsh) on the same matrix;
* the canonical basis does not depend on the basis it starts from: rotating each cluster's
  eigenvectors by a random orthogonal matrix (and flipping signs) leaves it unchanged; a simple
  eigenvalue's vector has a positive first non-vanishing entry;
* closed forms of the encoding: with the eigenvector column of W_{2->d_SPE} set to zero every
  node gets the same SPE; with zero query weights every attention row is uniform, so
  SPE_j = [mean lambda, mean_i phi_i[j]] W_pe (Wv_0 | ... | Wv_{h-1}) Wo, where
  mean lambda = 2|E| / T.
The host precompute (LAPACK eigensolver, an algebraic shortcut for the attention) agrees with
the oracle (Jacobi, the definition step by step) to 1e-8.
"""
import numpy as np
import pytest

from oracle import spe as OS
from paper_2410_05911_gb300 import inputs as I
from paper_2410_05911_gb300 import spe

CODES = [("hamming7_4", 8), ("bch31_16", 8), ("polar64_32", 16), ("bch63_36", 32), ("ldpc128_64", 32)]


@pytest.mark.parametrize("key", [c for c, _ in CODES])
def test_oracle_eigenpairs(key):
    H = I.make_code(key).H
    L = OS.laplacian(H)
    T = L.shape[0]
    # the Laplacian itself: symmetric, zero row sums, the degrees on the diagonal
    assert (L == L.T).all() and np.abs(L.sum(1)).max() == 0
    assert np.diag(L)[:H.shape[1]].tolist() == H.sum(0).tolist()
    lam, V, sweeps = OS.jacobi(L)
    assert sweeps < 100
    assert np.abs(L @ V - V * lam).max() < 1e-9
    assert np.abs(V.T @ V - np.eye(T)).max() < 1e-10
    assert abs(lam.sum() - 2 * H.sum()) < 1e-8
    assert np.abs(np.sort(lam) - np.linalg.eigvalsh(L)).max() < 1e-9
    lam_c, V_c = OS.canonical(lam, V)
    assert abs(lam_c[0]) < 1e-9 and lam_c[1] > 1e-6  # connected: one zero eigenvalue
    assert np.abs(V_c[:, 0] - 1.0 / np.sqrt(T)).max() < 1e-9  # the constant vector, positive


@pytest.mark.parametrize("key", ["hamming7_4", "ldpc128_64", "bch63_36"])
def test_canonical_basis_is_independent_of_the_starting_basis(key):
    H = I.make_code(key).H
    lam, V, _ = OS.jacobi(OS.laplacian(H))
    lam_c, V_c = OS.canonical(lam, V)
    rng = np.random.default_rng(3)
    # rotate every cluster of the canonical basis by a random orthogonal matrix, flip signs,
    # shuffle the columns: the canonical basis of the result must come back
    R = V_c.copy()
    T = lam_c.shape[0]
    tol = OS.CLUSTER_TOL * max(1.0, np.abs(lam_c).max())
    i = 0
    clusters = 0
    while i < T:
        j = i + 1
        while j < T and lam_c[j] - lam_c[j - 1] <= tol:
            j += 1
        Q, _ = np.linalg.qr(rng.standard_normal((j - i, j - i)))
        R[:, i:j] = V_c[:, i:j] @ (Q * rng.choice([-1.0, 1.0], j - i))
        clusters += j - i > 1
        i = j
    perm = rng.permutation(T)
    lam_r, V_r = OS.canonical(lam_c[perm], R[:, perm])
    assert np.abs(lam_r - lam_c).max() < 1e-12
    assert np.abs(V_r - V_c).max() < 1e-9
    if key == "ldpc128_64":
        assert clusters > 0  # the (3,6)-regular code has a repeated eigenvalue (3, on the null space of H)
    # a simple eigenvalue's vector: first entry above the vanishing threshold is positive
    for c in range(T):
        simple = (c == 0 or lam_c[c] - lam_c[c - 1] > tol) and (c == T - 1 or lam_c[c + 1] - lam_c[c] > tol)
        if simple:
            v = V_c[:, c]
            assert v[np.argmax(np.abs(v) > OS.VANISH_TOL)] > 0


def test_spe_without_eigenvector_column_is_the_same_for_every_node():
    H = I.make_code("bch31_16").H
    p = I.spe_params(H, 8, seed=11)
    p.w_pe[1] = 0.0
    out, _, _ = OS.table(H, p)
    assert np.abs(out - out[0]).max() < 1e-12
    assert np.abs(out[0]).max() > 1e-3


@pytest.mark.parametrize("key,d_spe", [("hamming7_4", 8), ("polar64_32", 16)])
def test_spe_with_uniform_attention_closed_form(key, d_spe):
    H = I.make_code(key).H
    p = I.spe_params(H, d_spe, seed=13)
    p.wq[:] = 0.0  # every score 0: softmax rows uniform
    out, lam, V = OS.table(H, p)
    T = lam.shape[0]
    assert abs(lam.mean() - 2 * H.sum() / T) < 1e-9
    mean_phi = V.sum(1) / T  # node j: mean over i of phi_i[j]
    Wv = np.concatenate(list(p.wv), 1)  # [d_spe, heads * d_e]
    want = (np.stack([np.full(T, lam.mean()), mean_phi], 1) @ p.w_pe) @ Wv @ p.wo
    assert np.abs(out - want).max() < 1e-10


@pytest.mark.parametrize("key,d_spe", CODES)
def test_host_precompute_matches_oracle(key, d_spe):
    H = I.make_code(key).H
    p = I.spe_params(H, d_spe, seed=5)
    ref, lam_o, V_o = OS.table(H, p)
    lam, U = spe.eigenpairs(H)
    assert np.abs(lam - lam_o).max() < 1e-9
    assert np.abs(U - V_o).max() < 1e-7
    got = spe.spe_from_eigenpairs(lam, U, p)
    assert np.abs(got - ref).max() < 1e-8 * (1.0 + np.abs(ref).max())
    # the float32 table the decoder takes
    tab = spe.spe_table(H, p)
    assert tab.dtype == np.float32 and np.abs(tab - ref).max() <= 1e-6 * (1.0 + np.abs(ref).max())


def test_workload_models_carry_the_laplacian_encoding():
    m = I.workload_model("bch31_16")
    p = I.spe_params(m.H, m.d_spe, seed=1000 + I.WORKLOADS["bch31_16"]["seed"] + 7919)
    ref, _, _ = OS.table(m.H, p)
    assert m.spe.shape == (m.n + m.n - m.k, m.d_spe)
    assert np.abs(m.spe - ref).max() <= 1e-6 * (1.0 + np.abs(ref).max())
