"""Full-precision linear layers (linear_mode = 1): the ECCT baseline of Sec. 3 (fp32 weights and
activations) in the tensor cores' bf16 format, decoded through the C ABI and compared with the
oracle.  The tensor cores accumulate in fp32 in an order of their own, so parity here is a bound,
not bit equality:

* block 0's Q, K, V sums, whose bf16 inputs are the same on both sides, agree with the oracle's
  exact sums rounded once to within the fp32 summation bound K 2^-23 sum_i |x_i w_i|;
* the logits agree within the float tolerance 2e-2 absolute, and the decoded bits are identical
  except where the oracle's logit is below 0.05 in magnitude, on at least 99.99% of the bits
  (each case decodes at least 10^4 bits);
* the syndromes are those of the decoded bits.
Also the ECCT configuration as a whole: GELU, the code-aware mask on every head (mask_mode 1)
and full-precision linears.
"""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2410_05911_gb300 import aecct as A
from paper_2410_05911_gb300 import inputs as I

torch = pytest.importorskip("torch")

CASES = [
    # (code, d, layers, variant, attention modes)
    ("bch31_16", 32, 2, dict(), (1, 2)),
    ("polar64_32", 64, 2, dict(), (1, 2)),
    ("ldpc128_64", 128, 2, dict(), (1,)),
    ("bch63_36", 128, 2, dict(), (1, 2)),
    ("bch31_16", 32, 2, dict(activation=1, mask_mode=1), (1, 2)),
    ("polar64_32", 64, 2, dict(activation=1, mask_mode=1), (2,)),
    ("bch63_36", 128, 1, dict(activation=1, mask_mode=1), (1,)),
]


def _block0_inputs(model, y):
    """fp32 block-0 input rows x[b][t] = [h_t emb_t, spe_t] (Sec. 3), computed here."""
    H = model.H.astype(np.int64)
    out = []
    for yb in y:
        s = (H @ (yb < 0).astype(np.int64)) % 2
        h = np.concatenate([np.abs(yb), (1.0 - 2.0 * s)]).astype(np.float32)
        out.append(np.concatenate([h[:, None] * model.emb, model.spe], 1).astype(np.float32))
    return np.stack(out)


@pytest.mark.gpu
@pytest.mark.parametrize("case", CASES, ids=[f"{c[0]}-{'-'.join(f'{k}{v}' for k, v in c[3].items()) or 'relu'}"
                                             for c in CASES])
def test_full_precision_linears(case):
    key, d, layers, var, modes = case
    code = I.make_code(key)
    var = dict(var)
    mask_mode = var.pop("mask_mode", 0)
    model = I.random_model(code, d, layers, seed=91, full_precision=True, **var)
    model.mask_mode = mask_mode
    B, capB = -(-10000 // code.n), 3
    y = I.channel_batch(code, B, 3.0, seed=7).y
    r = O.decode(model, y, cap_B=capB)
    ref = r["logits"].astype(np.float64)
    # block-0 QKV: |gpu - oracle| <= K 2^-23 sum_i |bf16(x_i) bf16(w_oi)|
    x0 = _block0_inputs(model, y[:capB])
    Wqkv = np.concatenate([np.asarray(w, np.float32) for w in model.w_full[0][:3]], 0)
    absprod = np.abs(O.bf16_round(x0).reshape(x0.shape)).astype(np.float64) @ \
        np.abs(O.bf16_round(Wqkv).reshape(Wqkv.shape)).astype(np.float64).T
    bound = d * 2.0 ** -23 * absprod + 1e-30
    want = r["capture"]["acc"][:, 0, 0, :, :3 * d].view(np.float32).astype(np.float64)
    for mode in modes:
        dec = A.Decoder(model, attention_mode=mode)
        cap = dec.set_capture(capB)
        bits, syn, logits = dec.decode(torch.from_numpy(y).cuda())
        torch.cuda.synchronize()
        assert dec.synchronize() == A.AECCT_OK
        got = cap["acc"].cpu().numpy()[:, 0, 0, :, :3 * d].view(np.float32).astype(np.float64)
        assert (np.abs(got - want) <= bound).all(), f"mode {mode}: block-0 sums outside the fp32 bound"
        lg = logits.cpu().numpy().astype(np.float64)
        diff = np.abs(lg - ref)
        assert diff.max() <= 2e-2, f"mode {mode}: max |d logit| {diff.max():.3e}, median {np.median(diff):.2e}"
        b = bits.cpu().numpy()
        flip = b != r["bits"]
        away = flip & (np.abs(ref) >= 0.05)
        assert away.mean() <= 1e-4, f"mode {mode}: {int(away.sum())} of {flip.size} bits differ where |logit| >= 0.05"
        assert (syn.cpu().numpy() == (b.astype(np.int64) @ model.H.T.astype(np.int64)) % 2).all()
        dec.close()
