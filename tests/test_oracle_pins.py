"""Pins for the CPU oracle against facts other than its own formulas.

Each test ties one oracle function to brute force, a closed form, a special case that
reduces to a textbook or library routine, or an exact invariance the paper states, so
that a dropped term, a wrong sign or index, or a transposed operand fails somewhere.
"""
import math

import networkx as nx
import numpy as np
import pytest

from oracle import oracle as O
from paper_2410_05911_gb300 import inputs as I

ALL_CODES = ["hamming7_4", "bch31_16", "polar64_32", "ldpc128_64", "bch63_36", "ldpc384_192"]


# ---------------------------------------------------------------------------
# canonical scalar pieces
# ---------------------------------------------------------------------------

def test_exp2_series_exact_at_integers():
    # f = 0 leaves only the constant term 1: 2^n must come out exactly
    xs = np.arange(-125, 1, dtype=np.float32)
    assert (O.exp2_series(xs) == np.exp2(xs.astype(np.float64)).astype(np.float32)).all()
    assert O.exp2_series([-126.0, -1e30])[0] == 0.0


def test_exp2_series_accuracy_vs_libm():
    rng = np.random.default_rng(0)
    xs = np.concatenate([-rng.uniform(0, 30, 4000), -rng.uniform(0, 1, 4000), [-0.5, -0.25, -1e-7, 0.0]])
    xs = xs.astype(np.float32)
    got = O.exp2_series(xs).astype(np.float64)
    ref = np.exp2(xs.astype(np.float64))
    ulp = np.spacing(ref.astype(np.float32)).astype(np.float64)
    assert (np.abs(got - ref) <= 2.0 * ulp).all()


def test_gelu_against_libm_erf():
    # GELU(x) = 0.5 x (1 + erf(x / sqrt 2)); the oracle's erf (Abramowitz & Stegun 7.1.26) is within
    # 1.5e-7 of erf, so GELU is within 0.5 |x| 1.5e-7 plus a few fp32 roundings of |x| and |GELU|
    rng = np.random.default_rng(3)
    xs = np.concatenate([np.linspace(-12, 12, 4001), rng.normal(0, 3, 4000)]).astype(np.float32)
    got = O.gelu(xs).astype(np.float64)
    x = xs.astype(np.float64)
    ref = np.array([0.5 * v * (1.0 + math.erf(v / math.sqrt(2.0))) for v in x])
    assert (np.abs(got - ref) <= 2.5e-7 * (np.abs(x) + np.abs(ref)) + 1e-45).all()


def test_gelu_special_values_and_odd_part():
    g = O.gelu([0.0, 30.0, -30.0, 100.0])
    assert g[0] == 0.0 and g[1] == 30.0 and g[2] == 0.0 and g[3] == 100.0
    # x Phi(x) - (-x) Phi(-x) = x Phi(x) + x (1 - Phi(x)) = x
    x = np.linspace(0.0, 10.0, 2001).astype(np.float32)
    d = O.gelu(x).astype(np.float64) - O.gelu(-x).astype(np.float64)
    assert (np.abs(d - x) <= 2e-7 * x + 1e-45).all()


def test_bf16_round_matches_torch_conversion():
    # round to nearest even to 8 significant bits: torch's fp32 -> bf16 conversion, with ties
    # (half an ulp exactly, odd and even kept parts) and values next to them
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(5)
    base = rng.standard_normal(3000).astype(np.float32)
    bits = base.view(np.uint32) & np.uint32(0xFFFF0000)
    ties = (bits | np.uint32(0x8000)).view(np.float32)
    x = np.concatenate([base, ties, np.nextafter(ties, np.float32(np.inf)), np.nextafter(ties, np.float32(-np.inf)),
                        np.float32([0.0, -0.0, 1.0, 65504.0, 1e-30, -3.0e38])]).astype(np.float32)
    want = torch.from_numpy(x).to(torch.bfloat16).to(torch.float32).numpy()
    assert (O.bf16_round(x).view(np.uint32) == want.view(np.uint32)).all()


def test_full_linear_row_is_the_exact_sum_rounded_once():
    # out_o - b_o = fp32 of the exact rational sum of bf16(x_i) bf16(W_oi)
    from fractions import Fraction
    rng = np.random.default_rng(6)
    K, N = 48, 7
    x = rng.uniform(-3, 3, K).astype(np.float32)
    W = (rng.standard_normal((N, K)) / 4).astype(np.float32)
    b = rng.standard_normal(N).astype(np.float32)
    s, out = O.full_linear_row(x, W, b)
    xb, Wb = O.bf16_round(x), O.bf16_round(W).reshape(N, K)
    assert not (xb == x).all()  # the rounding acts
    def nearest_f32(q):  # the fp32 value nearest to the rational q, ties to even
        c = np.float32(float(q))
        cands = [np.nextafter(c, np.float32(-np.inf)), c, np.nextafter(c, np.float32(np.inf))]
        return min(cands, key=lambda f: (abs(Fraction(float(f)) - q), int(np.float32(f).view(np.uint32)) & 1))

    for o in range(N):
        exact = sum(Fraction(float(xb[i])) * Fraction(float(Wb[o, i])) for i in range(K))
        assert s[o] == nearest_f32(exact)
        assert out[o] == np.float32(s[o] + b[o])


def test_exp2_series_coefficients_are_taylor_terms():
    c = O.exp2_coefficients()
    for kk in range(8):
        assert c[kk] == np.float32(math.log(2.0) ** kk / math.factorial(kk))


def test_pairwise_sum_order():
    # pairwise: (1e8 + 1) + (-1e8 + 1) -> 1e8 + (-1e8) = 0 in fp32; left-to-right would give 1
    v = np.array([1e8, 1.0, -1e8, 1.0], dtype=np.float32)
    assert O.psum(v) == np.float32(0.0)
    ints = np.arange(64, dtype=np.float32)
    assert O.psum(ints) == np.float32(64 * 63 / 2)


# ---------------------------------------------------------------------------
# S1 / S10: hard decision and syndrome
# ---------------------------------------------------------------------------

def test_hard_decision_signs():
    y = np.array([1.0, -1.0, 0.0, -0.0, 1e-30, -1e-30], dtype=np.float32)
    assert O.hard_decision(y).tolist() == [0, 1, 0, 0, 0, 1]


@pytest.mark.parametrize("key", ALL_CODES)
def test_syndrome_codeword_and_single_errors(key):
    c = I.make_code(key)
    ch = I.channel_batch(c, 4, 4.0, seed=1)
    for x in ch.codewords:
        assert not O.syndrome(c.H, x).any()
    # a single flipped bit j gives column j of H; syndromes are linear over GF(2)
    for j in range(0, c.n, max(1, c.n // 13)):
        e = np.zeros(c.n, np.uint8)
        e[j] = 1
        assert (O.syndrome(c.H, e) == c.H[:, j]).all()
        assert (O.syndrome(c.H, ch.codewords[0] ^ e) == c.H[:, j]).all()


# ---------------------------------------------------------------------------
# HPSA masks (Sec. 4.2) against graph distances in the Tanner graph
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("key", ["hamming7_4", "bch31_16", "polar64_32", "ldpc128_64", "bch63_36"])
def test_masks_match_tanner_distances(key):
    c = I.make_code(key)
    M1, M2 = O.masks(c.H)
    n, m = c.n, c.n - c.k
    G = nx.Graph()
    G.add_nodes_from(range(n + m))
    for i in range(m):
        for j in range(n):
            if c.H[i, j]:
                G.add_edge(j, n + i)
    dist = dict(nx.all_pairs_shortest_path_length(G, cutoff=2))
    T = n + m
    D = np.full((T, T), 99)
    for a, row in dist.items():
        for b, dd in row.items():
            D[a, b] = dd
    assert (M1 == (D == 1)).all()
    assert (M2 == ((D == 2) | (D == 0))).all()
    # 2|E| first-ring entries (App. A counts 2|E| d/2 multiplications for the first ring)
    assert M1.sum() == 2 * c.H.sum()
    assert (M1 == M1.T).all() and (M2 == M2.T).all()
    assert M1.sum(1).min() > 0 and M2.sum(1).min() > 0


def test_attention_sparsity_crosscheck():
    # Fig. 4: HPSA avoids >= 78% of query-key products for most codes (cross-check only)
    c = I.make_code("ldpc128_64")
    M1, M2 = O.masks(c.H)
    T = c.T
    hpsa = 1 - (4 * M1.sum() + 4 * M2.sum()) / (8 * T * T)
    assert hpsa > 0.9


# ---------------------------------------------------------------------------
# Sec. 4.1: activation quantiser, integer core, ternary quantiser
# ---------------------------------------------------------------------------

def test_quant_closed_forms():
    x = np.array([127.0, -127.0, 2.5, 3.5, -2.5, 0.49, 0.5, 0.51], dtype=np.float32)
    q, a = O.quant_row(x)
    assert a == np.float32(127.0)
    assert q.tolist() == [127, -127, 2, 4, -2, 0, 0, 1]  # r = 1: ties go to even
    q, a = O.quant_row(np.zeros(16, np.float32))
    assert a == np.float32(1e-5) and not q.any()
    x = np.array([0.5, -1.0, 0.25, 0.75], dtype=np.float32)
    q, a = O.quant_row(x)
    assert a == np.float32(1.0) and q.tolist() == [64, -127, 32, 95]  # 63.5 -> 64, 31.75 -> 32


def test_quant_invariants_random():
    rng = np.random.default_rng(3)
    for _ in range(200):
        x = (rng.standard_normal(64) * rng.uniform(0.01, 100)).astype(np.float32)
        q, a = O.quant_row(x)
        assert np.abs(q).max() == 127
        assert a == np.abs(x).max()
        # each code is within half a step of the scaled value (before the tie rule)
        r = np.float32(127.0) / a
        assert (np.abs(q - x * r) <= 0.5).all()
        # scaling the row by a power of two scales alpha and leaves the codes alone
        q2, a2 = O.quant_row(x * np.float32(8.0))
        assert (q2 == q).all() and a2 == a * 8


def test_aap_linear_bruteforce_integer_core():
    rng = np.random.default_rng(4)
    for K, N in [(8, 4), (64, 96), (256, 64)]:
        q = rng.integers(-127, 128, K).astype(np.int8)
        W = rng.integers(-1, 2, (N, K)).astype(np.int8)
        b = rng.standard_normal(N).astype(np.float32)
        acc, out = O.aap_linear_row(q, 2.0, W, 0.5, b)
        brute = [sum(int(q[i]) * int(W[o, i]) for i in range(K)) for o in range(N)]
        assert acc.tolist() == brute
        assert np.abs(acc).max() <= 127 * K
        f = np.float32(np.float32(0.5) * np.float32(2.0)) / np.float32(127.0)
        assert (out == (acc.astype(np.float32) * f + b).astype(np.float32)).all()
    # zero weights return the bias; identity weights return the codes times the scale
    q = rng.integers(-127, 128, 16).astype(np.int8)
    acc, out = O.aap_linear_row(q, 127.0, np.zeros((5, 16), np.int8), 1.0, np.arange(5, dtype=np.float32))
    assert not acc.any() and out.tolist() == [0, 1, 2, 3, 4]
    acc, out = O.aap_linear_row(q, 127.0, np.eye(16, dtype=np.int8), 1.0, np.zeros(16, np.float32))
    assert (acc == q).all() and (out == q.astype(np.float32)).all()


def test_ternary_quantizer_percentile_and_sparsity():
    rng = np.random.default_rng(5)
    W = rng.standard_normal(100001).astype(np.float32)
    t, sc = O.ternary(W, delta=2.0, eps=0.0)
    gamma = np.quantile(np.abs(W).astype(np.float64), 0.5)
    assert sc == pytest.approx(2.0 * gamma, rel=1e-6)
    assert set(np.unique(t)) <= {-1, 0, 1}
    # delta = 2: zero iff |W| < gamma, i.e. below the median of |W| -> half the weights
    assert (t == 0).mean() == pytest.approx(0.5, abs=2e-5)
    t1, _ = O.ternary(W, delta=1.0, eps=0.0)
    # delta = 1: zero iff |W| < gamma/2; for N(0,1): P(|W| < 0.6745/2) = 0.2644
    assert (t1 == 0).mean() == pytest.approx(0.2644, abs=0.005)
    assert ((t1 == np.sign(W)) | (t1 == 0)).all()
    # tiny worked case: |W| sorted = 0,1,2,3,4 -> median 2, delta 1 -> threshold at 1 (tie -> 0)
    t2, sc2 = O.ternary(np.array([0, -1, 2, -3, 4], np.float32), delta=1.0, eps=0.0)
    assert sc2 == 2.0 and t2.tolist() == [0, 0, 1, -1, 1]


# ---------------------------------------------------------------------------
# LayerNorm and attention
# ---------------------------------------------------------------------------

def test_layernorm_closed_forms():
    d = 64
    g = np.ones(d, np.float32)
    b = np.zeros(d, np.float32)
    rng = np.random.default_rng(6)
    v = (rng.standard_normal(d) * 3 + 1).astype(np.float32)
    y = O.layernorm_row(v, g, b, 1e-5)
    ref = (v - v.astype(np.float64).mean()) / np.sqrt(v.astype(np.float64).var() + 1e-5)
    assert np.abs(y - ref).max() < 1e-5
    # constant row -> beta; affine parameters applied per feature
    beta = np.arange(d, dtype=np.float32)
    assert (O.layernorm_row(np.full(d, 7.0, np.float32), g, beta) == beta).all()
    gam = np.linspace(0.5, 2, d).astype(np.float32)
    y2 = O.layernorm_row(v, gam, b)
    assert np.abs(y2 - ref * gam).max() < 1e-5


def test_attention_special_cases_and_dense_softmax():
    rng = np.random.default_rng(7)
    T, d, heads = 10, 16, 4
    M1 = (rng.uniform(size=(T, T)) < 0.3).astype(np.uint8)
    M2 = (rng.uniform(size=(T, T)) < 0.6).astype(np.uint8)
    M1[0] = 0
    M1[0, 3] = 1  # a row with one key
    M2[5] = 0
    M2[5, 5] = 1
    Q = rng.standard_normal((T, d)).astype(np.float32)
    K = rng.standard_normal((T, d)).astype(np.float32)
    V = rng.standard_normal((T, d)).astype(np.float32)
    A = O.attention(Q, K, V, heads, 2, M1, M2)
    dh = d // heads
    # single key -> exactly that key's value row
    assert (A[0, :dh] == V[3, :dh]).all()
    assert (A[5, 2 * dh:3 * dh] == V[5, 2 * dh:3 * dh]).all()
    # dense softmax with -inf masking in float64
    for e in range(heads):
        M = M1 if e < 2 else M2
        sl = slice(e * dh, (e + 1) * dh)
        s = Q[:, sl].astype(np.float64) @ K[:, sl].astype(np.float64).T / math.sqrt(dh)
        s = np.where(M > 0, s, -np.inf)
        has = M.sum(1) > 0
        s = s - np.where(has[:, None], s.max(1, keepdims=True), 0)
        p = np.where(M > 0, np.exp(s), 0)
        ref = np.where(has[:, None], (p @ V[:, sl].astype(np.float64)) / np.maximum(p.sum(1, keepdims=True), 1e-300), 0)
        assert np.abs(A[:, sl] - ref).max() < 1e-5
    # equal scores (K = 0) -> plain average of the neighbours' values
    A0 = O.attention(Q, np.zeros_like(K), V, heads, 2, M1, M2)
    e = 3
    sl = slice(e * dh, (e + 1) * dh)
    ref = (M2.astype(np.float64) @ V[:, sl]) / M2.sum(1, keepdims=True)
    assert np.abs(A0[:, sl] - ref).max() < 1e-6


# ---------------------------------------------------------------------------
# whole decoder
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("key", ["bch31_16", "polar64_32"])
def test_codeword_symmetry_invariance_exact(key):
    # Sec. 3: h(y) = [|y|, s(y)] is unchanged by y -> y * x_s(c) for a codeword c, so eps is
    # identical bit for bit, and the decoded word shifts by c
    w = I.workload(key)
    model = I.workload_model(key)
    ch = I.channel_batch(w.code, 6, 3.0, seed=9)
    r0 = O.decode(model, ch.y, nthreads=4)
    other = I.channel_batch(w.code, 6, 3.0, seed=10).codewords
    y2 = (ch.y * (1.0 - 2.0 * other.astype(np.float32))).astype(np.float32)
    r1 = O.decode(model, y2, nthreads=4)
    assert (r1["logits"].view(np.int32) == r0["logits"].view(np.int32)).all()
    assert ((r0["bits"] ^ other) == r1["bits"]).all()
    assert (r0["syndrome"] == r1["syndrome"]).all()


def _ln64(v, g, b, eps):
    mu = v.mean(-1, keepdims=True)
    var = ((v - mu) ** 2).mean(-1, keepdims=True)
    return (v - mu) / np.sqrt(var + eps) * g + b


def test_zero_weight_closed_form():
    # with every ternary weight zero each AAP layer returns its bias, attention averages
    # identical value rows, and a block maps x -> LN(LN(x + b_o) + b_2)
    code = I.make_code("bch31_16")
    model = I.random_model(code, 32, 3, seed=21, zero_weights=True)
    ch = I.channel_batch(code, 5, 2.0, seed=22)
    r = O.decode(model, ch.y, nthreads=2)
    y = ch.y.astype(np.float64)
    b = (y < 0).astype(np.int64)
    s = (b @ code.H.T.astype(np.int64)) % 2
    h = np.concatenate([np.abs(y), 1 - 2 * s], 1)
    de = model.d - model.d_spe
    x = np.concatenate([h[:, :, None] * model.emb[None], np.broadcast_to(model.spe[None], (5, code.T, model.d_spe))], 2)
    for l in range(model.n_layers):
        x = _ln64(x + model.bias[l][3], model.ln_gamma[l, 0], model.ln_beta[l, 0], model.ln_eps)
        x = _ln64(x + model.bias[l][5], model.ln_gamma[l, 1], model.ln_beta[l, 1], model.ln_eps)
    z = x @ model.w_d1.astype(np.float64) + model.b_d1
    eps = z @ model.w_out.astype(np.float64) + model.b_out
    assert np.abs(r["logits"] - eps).max() < 2e-4
    marg = np.abs(eps) < 1e-3
    assert ((r["bits"] == (y * eps < 0)) | marg).all()


def test_capture_integer_core_consistent():
    # every recorded accumulator row is the exact integer product of the recorded codes
    # and the model's ternary weights (Q,K,V stacked; O; FFN1; FFN2)
    key = "bch31_16"
    w = I.workload(key)
    model = I.workload_model(key)
    ch = I.channel_batch(w.code, 3, 4.0, seed=2)
    r = O.decode(model, ch.y, nthreads=1, cap_B=3)
    cap = r["capture"]
    d, F = model.d, 4 * model.d
    for l in range(model.n_layers):
        Wt = model.w_tern[l]
        for g, (Wm, K) in enumerate([(np.concatenate(Wt[0:3]), d), (Wt[3], d), (Wt[4], d), (Wt[5], F)]):
            q = cap["q"][:, l, g, :, :K].astype(np.int64)
            acc = cap["acc"][:, l, g, :, :Wm.shape[0]]
            assert (acc == q @ Wm.T.astype(np.int64)).all()
            assert (np.abs(q).max(-1) == 127).all() or g == 3
    # input syndrome record equals the syndrome of the hard decisions
    b = (ch.y < 0).astype(np.int64)
    assert (cap["syn_in"] == (b @ w.code.H.T.astype(np.int64)) % 2).all()
    # layer-0 QKV codes are Quant of the embedding rows
    s = cap["syn_in"][0].astype(np.float32)
    h = np.concatenate([np.abs(ch.y[0]), np.float32(1) - np.float32(2) * s]).astype(np.float32)
    de = d - model.d_spe
    for t in range(w.code.T):
        row = np.concatenate([(h[t] * model.emb[t]).astype(np.float32), model.spe[t]])
        q, a = O.quant_row(row)
        assert (cap["q"][0, 0, 0, t, :d] == q).all() and cap["alpha"][0, 0, 0, t] == a


def test_decode_validation_and_empty_batch():
    model = I.workload_model("bch31_16")
    r = O.decode(model, np.zeros((0, model.n), np.float32))
    assert r["bits"].shape == (0, model.n)
    bad = I.workload_model("bch31_16")
    bad.h_first = 9
    with pytest.raises(ValueError):
        O.decode(bad, np.zeros((1, bad.n), np.float32))
