"""The spectral positional encoding of Sec. 4.3 computed on the GPU (aecct_spe_table: parallel Jacobi
eigensolver in double precision, canonical eigenbasis, multi-head self-attention over the eigen-tokens,
average pooling) against the oracle's restatement (oracle/spe_oracle.c: cyclic Jacobi, the
definition step by step) and the package's host precompute, on every code of the workloads."""
import time

import numpy as np
import pytest

from oracle import spe as OS
from paper_2410_05911_gb300 import aecct as A
from paper_2410_05911_gb300 import inputs as I
from paper_2410_05911_gb300 import spe

pytest.importorskip("torch")

CODES = [("hamming7_4", 8), ("bch31_16", 8), ("polar64_32", 16), ("bch63_36", 32), ("ldpc128_64", 32),
         ("ldpc384_192", 32)]


@pytest.mark.gpu
@pytest.mark.parametrize("key,d_spe", CODES)
def test_gpu_spe_matches_oracle(key, d_spe):
    H = I.make_code(key).H
    p = I.spe_params(H, d_spe, seed=5)
    T = H.shape[0] + H.shape[1]
    t0 = time.perf_counter()
    tab, t64, lam, U = A.spe_table(H, p, want_eigen=True)
    dt = time.perf_counter() - t0
    # the oracle on every node (a sample of 16 for the 576-node code, whose O(T^3) attention it
    # evaluates node by node)
    nodes = np.arange(T) if T <= 200 else np.linspace(0, T - 1, 16).astype(np.int32)
    ref, lam_o, V_o = OS.table(H, p, nodes)
    assert np.abs(lam - lam_o).max() < 1e-9
    assert np.abs(U - V_o).max() < 1e-7
    scale = 1.0 + np.abs(ref).max()
    assert np.abs(t64[nodes] - ref).max() < 1e-8 * scale
    assert np.abs(tab[nodes].astype(np.float64) - ref).max() <= 1e-6 * scale
    # and the host precompute of the package, on every node
    host = spe.spe_table(H, p)
    assert np.abs(tab - host).max() <= 2e-6 * (1.0 + np.abs(host).max())
    print(f"{key}: T = {T}, GPU SPE precompute {1e3 * dt:.1f} ms")
