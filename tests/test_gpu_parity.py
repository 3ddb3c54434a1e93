"""Parity of the CUDA decoder (through the C ABI) with the CPU oracle.

Both sides follow the same fp32 operation order, so the comparison is exact: logits
bit for bit, decoded bits, syndromes, and every recorded int8 code, alpha and int32
accumulator of every block.  Exactness implies the looser bars (|d logit| <= 2e-2,
bits identical except where |logit| < 0.05 on >= 99.99% of bits).
"""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2410_05911_gb300 import aecct as A
from paper_2410_05911_gb300 import inputs as I

torch = pytest.importorskip("torch")

KEYS = ["bch31_16", "polar64_32", "ldpc128_64", "bch63_36", "ldpc384_192"]
SMALL_B = {"bch31_16": 61, "polar64_32": 23, "ldpc128_64": 5, "bch63_36": 15, "ldpc384_192": 3}
SAMPLE_B = {"bch31_16": 64, "polar64_32": 48, "ldpc128_64": 12, "bch63_36": 24, "ldpc384_192": 6}

_decoders = {}


def decoder(key, cluster_ctas=0, attention_mode=0):
    k = (key, cluster_ctas, attention_mode)
    if k not in _decoders:
        _decoders[k] = (A.Decoder(I.workload_model(key), cluster_ctas=cluster_ctas, attention_mode=attention_mode),
                        I.workload_model(key))
    return _decoders[k]


def gpu_decode(dec, y, cap_B=0):
    cap = dec.set_capture(cap_B) if cap_B else dec.set_capture(0)
    yt = torch.from_numpy(y).cuda()
    bits, syn, logits = dec.decode(yt)
    torch.cuda.synchronize()
    assert dec.synchronize() == A.AECCT_OK
    out = dict(bits=bits.cpu().numpy(), syndrome=syn.cpu().numpy(), logits=logits.cpu().numpy())
    if cap is not None:
        out["capture"] = {k: v.cpu().numpy() for k, v in cap.items()}
        dec.set_capture(0)
    return out


def assert_same(g, r, label=""):
    dl = np.abs(g["logits"].astype(np.float64) - r["logits"])
    msg = f"{label}: max|dlogit| {dl.max():.3e}, logits differ at {(g['logits'] != r['logits']).sum()} places"
    assert (g["logits"].view(np.int32) == r["logits"].view(np.int32)).all(), msg
    assert (g["bits"] == r["bits"]).all(), label
    assert (g["syndrome"] == r["syndrome"]).all(), label


@pytest.mark.gpu
@pytest.mark.parametrize("key", KEYS)
def test_small_batch_exact_with_integer_core(key):
    dec, model = decoder(key)
    w = I.workload(key)
    B = SMALL_B[key]
    ch = I.channel_batch(w.code, B, w.ebn0_db[0], seed=100 + B)
    cap_B = min(B, 3)
    g = gpu_decode(dec, ch.y, cap_B=cap_B)
    r = O.decode(model, ch.y, cap_B=cap_B)
    for name in ("syn_in", "q", "alpha", "acc"):
        a, b = g["capture"][name], r["capture"][name]
        if name == "alpha":
            a, b = a.view(np.int32), b.view(np.int32)
        bad = np.argwhere(a != b)
        # index layout: [word, block, gemm (0 QKV, 1 O, 2 FFN1, 3 FFN2), token, column]
        assert bad.size == 0, (f"{name}: {len(bad)} entries differ, first at {bad[:4].tolist()} "
                               f"(gpu {a[tuple(bad[0])]} oracle {b[tuple(bad[0])]})")
    assert_same(g, r, key)


LAYOUTS = {
    # (cluster_ctas, attention_mode): per-row lists over a packed cluster, one CTA per group,
    # warp tasks (one CTA per group; at d = 128 with Q and A in TMEM and the checks' rows from the
    # next 32-row boundary), per-row lists over per-head staged rows (d = 128; one CTA or a cluster)
    "bch31_16": [(0, 1), (1, 1), (0, 2)],
    "polar64_32": [(0, 1), (1, 1), (0, 2)],
    "bch63_36": [(0, 1), (1, 1), (0, 2), (2, 1), (0, 3), (1, 3), (2, 3)],
    "ldpc128_64": [(0, 1), (0, 3), (2, 3), (4, 3)],
    "ldpc384_192": [(0, 1), (0, 3), (6, 3)],
}


@pytest.mark.gpu
@pytest.mark.parametrize("key", sorted(LAYOUTS))
def test_result_independent_of_layout_and_attention_mode(key):
    w = I.workload(key)
    ch = I.channel_batch(w.code, 40 if w.code.T <= 192 else 12, w.ebn0_db[-1], seed=77)
    ref = O.decode(I.workload_model(key), ch.y)
    for cc, mode in LAYOUTS[key]:
        dec, _ = decoder(key, cluster_ctas=cc, attention_mode=mode)
        q = dec.query()
        assert q["attention_mode"] == mode and (cc == 0 or q["cluster_ctas"] == cc)
        assert_same(gpu_decode(dec, ch.y), ref, f"{key} C={q['cluster_ctas']} mode={mode}")


@pytest.mark.gpu
@pytest.mark.parametrize("key", ["bch63_36", "ldpc128_64", "ldpc384_192"])
def test_staged_cluster_size_holds_the_most_words(key):
    # staged attention with the cluster size left open takes the size with the most words
    # resident on the device (words per group x clusters that fit at once)
    model = I.workload_model(key)
    dec = A.Decoder(model, attention_mode=3)
    q = dec.query()
    dec.close()
    best = q["words_per_group"] * q["max_clusters"]
    for c in range(1, 9):
        try:
            d2 = A.Decoder(model, cluster_ctas=c, attention_mode=3)
        except A.AecctError:
            continue  # no word fits, or the group passes the staged row limit
        q2 = d2.query()
        d2.close()
        assert q2["words_per_group"] * q2["max_clusters"] <= best, (c, q2, q)


@pytest.mark.gpu
@pytest.mark.parametrize("key", ["bch31_16", "polar64_32", "ldpc128_64"])
def test_codeword_symmetry_invariance_gpu(key):
    dec, model = decoder(key)
    w = I.workload(key)
    ch = I.channel_batch(w.code, 33, 3.0, seed=5)
    other = I.channel_batch(w.code, 33, 3.0, seed=6).codewords
    y2 = (ch.y * (1.0 - 2.0 * other.astype(np.float32))).astype(np.float32)
    a = gpu_decode(dec, ch.y)
    b = gpu_decode(dec, y2)
    assert (a["logits"].view(np.int32) == b["logits"].view(np.int32)).all()
    assert ((a["bits"] ^ other) == b["bits"]).all()
    assert (a["syndrome"] == b["syndrome"]).all()


@pytest.mark.gpu
@pytest.mark.parametrize("key", KEYS)
def test_full_size_batch_sampled_exact(key):
    # the workload at its full batch size, in the launch configuration the benchmark uses;
    # the oracle recomputes sampled words one by one, the syndrome property is checked on all
    dec, model = decoder(key)
    w = I.workload(key)
    ch = I.channel_batch(w.code, w.batch, w.ebn0_db[0], seed=2024)
    g = gpu_decode(dec, ch.y)
    rng = np.random.default_rng(1)
    S = SAMPLE_B[key]
    idx = np.unique(np.concatenate([[0, w.batch - 1], rng.choice(w.batch, S - 2, replace=False)]))
    r = O.decode(model, ch.y[idx])
    sub = {k: v[idx] for k, v in g.items()}
    assert_same(sub, r, key)
    Hm = w.code.H.astype(np.int64)
    assert (g["syndrome"] == (g["bits"].astype(np.int64) @ Hm.T) % 2).all()
    # decoding statistics are only reported: synthetic weights carry no trained meaning


POINTS = [(key, e) for key in KEYS for e in I.workload(key).ebn0_db]


@pytest.mark.gpu
@pytest.mark.parametrize("key,ebn0", POINTS, ids=[f"{k}-{e}dB" for k, e in POINTS])
def test_every_ebn0_point_against_oracle(key, ebn0):
    # at least 10^4 bits per configuration point (so that the 99.99% decision rule is measurable),
    # in the default launch configuration: bit-exact logits, decisions and syndromes, which meet
    # the float criteria (|d logit| <= 2e-2, decisions equal where |logit| >= 0.05) with margin
    dec, model = decoder(key)
    w = I.workload(key)
    B = -(-10000 // w.code.n)
    ch = I.channel_batch(w.code, B, ebn0, seed=9000 + int(10 * ebn0))
    g = gpu_decode(dec, ch.y)
    r = O.decode(model, ch.y)
    assert g["bits"].size >= 10000
    dl = np.abs(g["logits"].astype(np.float64) - r["logits"])
    assert dl.max() <= 2e-2
    differ = g["bits"] != r["bits"]
    assert (differ & (np.abs(r["logits"]) >= 0.05)).mean() <= 1e-4
    assert_same(g, r, f"{key} {ebn0} dB")


@pytest.mark.gpu
def test_edge_batches_and_optional_outputs():
    dec, model = decoder("polar64_32")
    w = I.workload("polar64_32")
    # B = 0 is a no-op
    y0 = torch.zeros((0, w.code.n), dtype=torch.float32, device="cuda")
    bits, syn, logits = dec.decode(y0)
    assert bits.shape == (0, w.code.n)
    # B = 1 and a ragged tail (B not a multiple of the words per group)
    for B in (1, 2, 5, 7):
        ch = I.channel_batch(w.code, B, 5.0, seed=B)
        g = gpu_decode(dec, ch.y)
        r = O.decode(model, ch.y)
        assert_same(g, r, f"B={B}")
    # without syndrome and logits outputs the bits are unchanged
    ch = I.channel_batch(w.code, 9, 5.0, seed=9)
    yt = torch.from_numpy(ch.y).cuda()
    b1, s1, l1 = dec.decode(yt, want_syndrome=False, want_logits=False)
    b2, _, _ = dec.decode(yt)
    torch.cuda.synchronize()
    assert s1 is None and l1 is None and torch.equal(b1, b2)
    # all-zero channel output (every |y| = 0, every hard decision 0) and huge magnitudes
    big = np.where(np.arange(4 * w.code.n).reshape(4, -1) % 3 == 0, -1e6, 1e6).astype(np.float32)
    for y in (np.zeros((4, w.code.n), np.float32), big):
        g = gpu_decode(dec, y)
        r = O.decode(model, y)
        assert_same(g, r, "extreme y")
    with pytest.raises(ValueError):
        dec.decode(yt.double())


@pytest.mark.gpu
def test_host_buffer_entry_point():
    dec, model = decoder("bch31_16")
    w = I.workload("bch31_16")
    ch = I.channel_batch(w.code, 100, 4.0, seed=3)
    bits, syn, logits = dec.decode_host(ch.y)
    r = O.decode(model, ch.y)
    assert_same(dict(bits=bits, syndrome=syn, logits=logits), r, "host")


@pytest.mark.gpu
@pytest.mark.parametrize("label,make,d,layers,B", [
    # the smallest code: 12 ten-token words per CTA, a batch that leaves a ragged last group
    ("hamming7_4", lambda: I.make_code("hamming7_4"), 32, 2, 31),
    # the largest token count this build takes: T = 1020 tokens over a cluster of 8 CTAs
    ("ldpc680_340", lambda: I.ldpc_regular_code(680, 340, 3, 6, seed=680340), 32, 1, 3),
    ("ldpc680_340-d64", lambda: I.ldpc_regular_code(680, 340, 3, 6, seed=680340), 64, 1, 2),
])
def test_extreme_shapes_exact(label, make, d, layers, B):
    code = make()
    model = I.random_model(code, d, layers, seed=17, spe_noise=code.T > 600)
    dec = A.Decoder(model)
    q = dec.query()
    if code.T > 896:
        assert q["cluster_ctas"] == 8
    ch = I.channel_batch(code, B, 3.0, seed=19)
    g = gpu_decode(dec, ch.y, cap_B=min(B, 2))
    r = O.decode(model, ch.y, cap_B=min(B, 2))
    assert_same(g, r, label)
    for name in ("q", "acc", "alpha", "syn_in"):
        a, b = g["capture"][name], r["capture"][name]
        assert (a.view(np.int32) if a.dtype == np.float32 else a).tolist() == \
            (b.view(np.int32) if b.dtype == np.float32 else b).tolist(), f"{label}: {name}"
    dec.close()


@pytest.mark.gpu
@pytest.mark.parametrize("label,make,d,layers,B", [
    # d = 128 warp tasks: the variables start at row 0 and the checks at the next 32-row boundary,
    # so the rows per word Tp run from 35 (more padding than tokens) to the limit 128
    ("hamming7_4", lambda: I.make_code("hamming7_4"), 128, 2, 13),
    ("bch31_16", lambda: I.make_code("bch31_16"), 128, 1, 11),
    ("polar64_32", lambda: I.make_code("polar64_32"), 128, 1, 7),
    ("ldpc96_64", lambda: I.ldpc_regular_code(96, 64, 3, 9, seed=9664), 128, 1, 5),
    # d <= 64 warp tasks pack the tokens: T = 126 of the 128 rows of a CTA
    ("ldpc98_70", lambda: I.ldpc_regular_code(98, 70, 2, 7, seed=0), 64, 2, 6),
    ("ldpc98_70-d32", lambda: I.ldpc_regular_code(98, 70, 2, 7, seed=0), 32, 1, 6),
])
def test_warp_tasks_row_limits_exact(label, make, d, layers, B):
    code = make()
    model = I.random_model(code, d, layers, seed=23)
    ch = I.channel_batch(code, B, 3.0, seed=29)
    r = O.decode(model, ch.y, cap_B=min(B, 3))
    smem = {}
    for mode in ((1, 2, 3) if d == 128 else (1, 2)):
        dec = A.Decoder(model, attention_mode=mode)
        q = dec.query()
        assert q["attention_mode"] == mode
        smem[mode] = q["smem_bytes"]
        g = gpu_decode(dec, ch.y, cap_B=min(B, 3))
        assert_same(g, r, f"{label} mode {mode}")
        for name in ("q", "acc", "alpha", "syn_in"):
            a, b = g["capture"][name], r["capture"][name]
            assert (a.view(np.int32) if a.dtype == np.float32 else a).tolist() == \
                (b.view(np.int32) if b.dtype == np.float32 else b).tolist(), f"{label} mode {mode}: {name}"
        dec.close()
    if d == 128:  # Q stays in TMEM: every mode lays out shared memory alike (tasks add their plan)
        assert smem[1] == smem[3] and 0 < smem[2] - smem[1] <= 8192


@pytest.mark.gpu
@pytest.mark.parametrize("key", ["bch31_16", "polar64_32", "bch63_36"])
def test_non_finite_word_leaves_the_others_exact(key):
    # a NaN or infinity in one word reaches only that word's rows (every step is row-local or
    # within one word), so the other words of the batch, including one sharing its CTA, decode
    # exactly as without it
    dec, model = decoder(key)
    w = I.workload(key)
    ch = I.channel_batch(w.code, 6, 4.0, seed=41)
    y = ch.y.copy()
    y[2, 0] = np.nan  # BCH(31,16) packs two words per CTA: words 3 and 4 share a CTA with these
    y[5, 1] = -np.inf
    g = gpu_decode(dec, y)
    keep = [0, 1, 3, 4]
    r = O.decode(model, ch.y[keep])
    assert_same({k: v[keep] for k, v in g.items()}, r, key)
