"""Model variants the paper discusses beyond its main configuration, decoded through the C ABI
and compared bit for bit with the oracle (every int8 code, alpha and int32 accumulator of every
block, then logits, bits and syndromes):

* the split of heads between the first-ring and second-ring masks (Sec. 4.2 uses half and
  half; App. C discusses other splits): h_first = 2 and 6 of 8 heads;
* binary weights in {-1, +1} (App. D) in place of ternary ones, through the same 2-bit format;
* the ECCT code-aware mask (Sec. 3; the CASA baseline the paper compares HPSA with): every head
  attends over the union of the two rings (mask_mode = 1);
* one absmax alpha per quantised matrix of a word instead of per token (alpha_mode = 1, the
  other reading of Sec. 4.1's scalar alpha of x);
* GELU in place of ReLU in the feed-forward block (activation = 1), whose output can be negative.
"""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2410_05911_gb300 import aecct as A
from paper_2410_05911_gb300 import inputs as I

torch = pytest.importorskip("torch")

CASES = [
    # (code, d, layers, variant, attention modes to run)
    ("bch31_16", 32, 2, dict(h_first=2), (1, 2)),
    ("bch31_16", 32, 2, dict(h_first=6), (1, 2)),
    ("polar64_32", 64, 2, dict(h_first=2), (1, 2)),
    ("polar64_32", 64, 2, dict(binary=True), (2,)),
    ("bch31_16", 32, 2, dict(binary=True, h_first=6), (1, 2)),
    ("ldpc128_64", 128, 2, dict(h_first=6), (1,)),
    ("bch63_36", 128, 1, dict(binary=True), (1, 2)),
    ("bch31_16", 32, 2, dict(mask_mode=1), (1, 2)),
    ("polar64_32", 64, 2, dict(mask_mode=1), (1, 2)),
    ("ldpc128_64", 128, 1, dict(mask_mode=1), (1,)),
    ("bch31_16", 32, 2, dict(alpha_mode=1), (1, 2)),
    ("polar64_32", 64, 2, dict(alpha_mode=1), (1, 2)),
    ("bch63_36", 128, 1, dict(alpha_mode=1, mask_mode=1), (1,)),
    ("bch31_16", 32, 2, dict(activation=1), (1, 2)),
    ("polar64_32", 64, 2, dict(activation=1), (1, 2)),
    ("ldpc128_64", 128, 1, dict(activation=1), (1,)),
    ("bch63_36", 128, 2, dict(activation=1, alpha_mode=1), (1,)),
    ("bch63_36", 128, 2, dict(activation=1, h_first=2), (1, 2)),
    ("bch63_36", 128, 1, dict(mask_mode=1), (1, 2)),
    ("bch63_36", 128, 1, dict(h_first=6), (1, 2, 3)),
    ("bch63_36", 128, 1, dict(h_first=1), (2, 3)),
]


def _capture_equal(g, r):
    for name in ("syn_in", "q", "alpha", "acc"):
        a, b = g[name], r[name]
        if name == "alpha":
            a, b = a.view(np.int32), b.view(np.int32)
        bad = np.argwhere(a != b)
        assert bad.size == 0, f"{name}: {len(bad)} entries differ, first at {bad[:4].tolist()}"


@pytest.mark.gpu
@pytest.mark.parametrize("case", CASES, ids=[f"{c[0]}-{'-'.join(f'{k}{v}' for k, v in c[3].items())}" for c in CASES])
def test_variant_exact(case):
    key, d, layers, var, modes = case
    code = I.make_code(key)
    var = dict(var)
    mask_mode = var.pop("mask_mode", 0)
    alpha_mode = var.pop("alpha_mode", 0)
    model = I.random_model(code, d, layers, seed=77, zero_frac=0.5, **var)
    model.mask_mode = mask_mode
    model.alpha_mode = alpha_mode
    if var.get("binary"):
        assert all((np.abs(t) == 1).all() for wl in model.w_tern for t in wl)
    B = 9
    y = I.channel_batch(code, B, 3.0, seed=5).y
    r = O.decode(model, y, cap_B=3)
    for mode in modes:
        dec = A.Decoder(model, attention_mode=mode)
        cap = dec.set_capture(3)
        bits, syn, logits = dec.decode(torch.from_numpy(y).cuda())
        torch.cuda.synchronize()
        assert dec.synchronize() == A.AECCT_OK
        _capture_equal({k: v.cpu().numpy() for k, v in cap.items()}, r["capture"])
        assert (logits.cpu().numpy().view(np.int32) == r["logits"].view(np.int32)).all(), f"mode {mode}"
        assert (bits.cpu().numpy() == r["bits"]).all() and (syn.cpu().numpy() == r["syndrome"]).all()
        dec.close()
