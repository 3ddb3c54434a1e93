"""Pins for the seeded input generators (code constructions, channel, synthetic weights).

These check the problem instances against textbook facts: G H^T = 0 over GF(2), the
BCH designed distance by brute force, the Arikan kernel identity G_N G_N = I, LDPC
regularity, and the AWGN noise level.
"""
import itertools
import math

import numpy as np
import pytest

from paper_2410_05911_gb300 import inputs as I

CODES = ["bch31_16", "polar64_32", "ldpc128_64", "bch63_36", "ldpc384_192", "hamming7_4"]


@pytest.mark.parametrize("key", CODES)
def test_generator_parity_orthogonal(key):
    # Sec. 3: G H^T = 0 over GF(2); every encoded codeword satisfies H x = 0
    c = I.make_code(key)
    assert not ((c.G.astype(np.int64) @ c.H.T.astype(np.int64)) % 2).any()
    assert c.H.shape == (c.n - c.k, c.n)
    assert set(np.unique(c.H)) <= {0, 1}
    ch = I.channel_batch(c, 257, 4.0, seed=11)
    assert not ((ch.codewords.astype(np.int64) @ c.H.T.astype(np.int64)) % 2).any()


@pytest.mark.parametrize("key,k_expected,T", [("bch31_16", 16, 46), ("bch63_36", 36, 90), ("polar64_32", 32, 96),
                                            ("ldpc128_64", 64, 192), ("ldpc384_192", 192, 576)])
def test_dimensions_and_token_count(key, k_expected, T):
    c = I.make_code(key)
    assert c.k == k_expected
    assert c.T == T  # 2n - k tokens
    assert I.gf2_rank(c.H) == c.n - c.k or key.startswith("ldpc")
    assert c.G.shape[0] == c.n - I.gf2_rank(c.H)


def test_bch31_minimum_distance_bruteforce():
    # designed distance 2t+1 = 7; a narrow-sense BCH(31,16) has d_min = 7
    c = I.make_code("bch31_16")
    msgs = np.array(list(itertools.product([0, 1], repeat=c.k)), dtype=np.int64)
    cw = (msgs @ c.G.astype(np.int64)) % 2
    w = cw.sum(1)
    assert w[1:].min() == 7
    assert c.n - c.k == 15  # deg g(x) = 15


def test_bch63_degree_and_cyclic():
    c = I.make_code("bch63_36")
    assert c.n - c.k == 27  # deg g(x) = 6+6+6+6+3 (coset of 9 has size 3)
    # cyclic: a cyclic shift of a codeword is a codeword
    ch = I.channel_batch(c, 64, 5.0, seed=3)
    sh = np.roll(ch.codewords, 1, axis=1)
    assert not ((sh.astype(np.int64) @ c.H.T.astype(np.int64)) % 2).any()


def test_bch63_low_weight_codewords_respect_designed_distance():
    # no codeword of weight < 11 among sums of up to 3 generator rows (spot check of d >= 11)
    c = I.make_code("bch63_36")
    G = c.G.astype(np.int64)
    for r in range(1, 4):
        for comb in itertools.combinations(range(c.k), r):
            if r == 3 and comb[0] > 4:
                break
            w = (G[list(comb)].sum(0) % 2).sum()
            assert w >= 11


def test_polar_kernel_and_frozen_set():
    c = I.make_code("polar64_32")
    GN = c.GN
    assert not ((GN.astype(np.int64) @ GN.astype(np.int64)) % 2 - np.eye(64, dtype=np.int64)).any()
    assert len(c.frozen) == 32
    # H = G_N[:, frozen]^T
    assert (c.H == GN[:, c.frozen].T).all()
    # bit-channel 0 is the worst channel and the last one is the best: 0 frozen, 63 not
    assert 0 in c.frozen and 63 not in c.frozen
    # Bhattacharyya recursion keeps the polarisation order: frozen indices have Z >= info indices
    z = [math.exp(-0.5)]
    while len(z) < 64:
        z = [2 * v - v * v for v in z] + [v * v for v in z]
    info = [j for j in range(64) if j not in c.frozen]
    assert min(z[j] for j in c.frozen) >= max(z[j] for j in info)


@pytest.mark.parametrize("key", ["ldpc128_64", "ldpc384_192"])
def test_ldpc_regular(key):
    c = I.make_code(key)
    assert (c.H.sum(0) == 3).all()
    assert (c.H.sum(1) == 6).all()
    assert c.H.max() == 1  # no repeated edge survives as a 2


def test_awgn_sigma_and_bpsk():
    assert I.awgn_sigma(0.0, 0.5) == pytest.approx(1.0)
    assert I.awgn_sigma(10 * math.log10(2.0), 0.5) == pytest.approx(1 / math.sqrt(2))
    c = I.make_code("polar64_32")
    ch = I.channel_batch(c, 20000, 3.0, seed=5)
    noise = ch.y - (1.0 - 2.0 * ch.codewords)
    assert noise.std() == pytest.approx(I.awgn_sigma(3.0, 0.5), rel=0.01)
    assert abs(noise.mean()) < 0.01


def test_synthetic_weights_zero_fraction_and_values():
    m = I.workload_model("polar64_32")
    for layer in m.w_tern:
        for t in layer:
            assert set(np.unique(t)) <= {-1, 0, 1}
            assert (t == 0).mean() == pytest.approx(0.4, abs=1.0 / t.size)
    m2 = I.workload_model("ldpc128_64")
    assert (m2.w_tern[0][0] == 0).mean() == pytest.approx(0.5, abs=1e-4)
    # 12 d^2 N linear weights; the paper's largest ECCT has about 2M parameters
    m3 = I.workload_model("bch63_36")
    assert sum(t.size for layer in m3.w_tern for t in layer) == 12 * 128 * 128 * 10 == 1966080


def test_ternary_scale_constant():
    # half-scale threshold at the median of |N(0, s^2)| gives 50% zeros: scale = 2 * 0.6745 s
    assert I.ternary_scale_for_zero_fraction(0.5, 64) == pytest.approx(2 * 0.67449 / 8, rel=1e-4)


def test_binary_weight_variant():
    code = I.make_code("bch31_16")
    m = I.random_model(code, 32, 2, seed=3, binary=True)
    for l in range(2):
        for g, t in enumerate(m.w_tern[l]):
            assert set(np.unique(t).tolist()) == {-1, 1}
            d_in = t.shape[1]
            base = np.sqrt(2.0 / (np.pi * d_in))
            assert 0.9 * base - 1e-7 <= m.w_scale[l, g] <= 1.1 * base + 1e-7
