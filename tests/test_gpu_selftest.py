"""GPU diagnostics: the tcgen05 MMA path on one tile, and the bounded device-side wait."""
import numpy as np
import pytest

from paper_2410_05911_gb300 import aecct as A


@pytest.mark.gpu
@pytest.mark.parametrize("K,N", [(16, 16), (32, 96), (64, 64), (64, 128), (128, 256), (128, 32)])
def test_tcgen05_mma_matches_integer_product(K, N):
    rng = np.random.default_rng(K * 1000 + N)
    a = rng.integers(-127, 128, (128, K)).astype(np.int8)
    b = rng.integers(-1, 2, (N, K)).astype(np.int8)
    out = A.selftest_mma(a, b)
    ref = a.astype(np.int64) @ b.T.astype(np.int64)
    assert (out == ref).all(), f"max |diff| {np.abs(out - ref).max()}"


@pytest.mark.gpu
def test_bounded_wait_reports_timeout():
    # the barrier is never completed: the wait must give up by itself and say so
    assert A.selftest_timeout(1 << 20) == A.AECCT_ERR_TIMEOUT
