"""The GPU against a float64 forward pass that was not written with the kernel in mind.

The CUDA decoder and the oracle follow one fixed fp32 order of operations, so their bit-for-bit
agreement shows that two implementations of that order agree.  This file checks the GPU on its
own against the paper's definitions: the float64 pass of `f64_forward` (numpy, written from
Sec. 3, 4.1-4.3 and 5, sharing nothing with either implementation) is teacher-forced on the
integer core the GPU itself recorded (int8 codes, alpha and int32 accumulators of every GEMM of
every block, through aecct_set_capture), and checks that

* every GPU alpha is max(|x|, floor) of the float64 input row and every GPU int8 code equals
  rint(x * 127 / alpha) of it, except at a rounding boundary (eq. Quant);
* the GPU logits are within 2e-2 absolute of the float64 logits;
* the GPU's decisions equal [y * eps < 0] of the float64 logits, except where |eps| < 0.05, on
  at least 99.99% of the bits.
A code may differ from the float64 rounding only within 1e-3 of a rounding boundary, and such
codes are rare: fp32 and float64 inputs differ by a few fp32 ulps, so about one code in 10^5
lands within that distance of a half-integer (the bound allows 10^-5 of the codes checked).

All five workloads at their real width d and depth N, at every Eb/N0 point they name.
"""
import numpy as np
import pytest

from f64_forward import forward64
from paper_2410_05911_gb300 import aecct as A
from paper_2410_05911_gb300 import inputs as I

torch = pytest.importorskip("torch")

POINTS = [(key, e) for key in ["bch31_16", "polar64_32", "ldpc128_64", "bch63_36", "ldpc384_192"]
          for e in I.workload(key).ebn0_db]
_decoders = {}


def _decoder(key):
    if key not in _decoders:
        _decoders[key] = A.Decoder(I.workload_model(key))
    return _decoders[key]


@pytest.mark.gpu
@pytest.mark.parametrize("key,ebn0", POINTS, ids=[f"{k}-{e}dB" for k, e in POINTS])
def test_gpu_capture_matches_float64_forward(key, ebn0):
    w = I.workload(key)
    model = I.workload_model(key)
    dec = _decoder(key)
    B = 3
    y = I.channel_batch(w.code, B, ebn0, seed=4000 + int(10 * ebn0)).y
    cap = dec.set_capture(B)
    bits, syn, logits = dec.decode(torch.from_numpy(y).cuda())
    torch.cuda.synchronize()
    assert dec.synchronize() == A.AECCT_OK
    capture = {k: v.cpu().numpy() for k, v in cap.items()}
    dec.set_capture(0)
    # the GPU's input syndromes are those of its channel outputs (Sec. 3)
    s_ref = (w.code.H.astype(np.int64) @ (y < 0).astype(np.int64).T).T % 2
    assert (capture["syn_in"] == s_ref).all()
    ref, boundary = forward64(model, y, capture)
    T, d = w.code.T, model.d
    codes = B * model.n_layers * T * (3 * d + 4 * d)  # the inputs of QKV, O, FFN1 (K = d) and FFN2 (K = 4d)
    assert boundary <= max(2, 1e-5 * codes), f"{boundary} of {codes} codes at a rounding boundary"
    g = logits.cpu().numpy().astype(np.float64)
    dl = np.abs(g - ref)
    assert dl.max() <= 2e-2, f"max |d logit| {dl.max():.3e}"
    want = (y.astype(np.float64) * ref < 0).astype(np.uint8)
    differ = bits.cpu().numpy() != want
    assert (differ & (np.abs(ref) >= 0.05)).mean() <= 1e-4, "decisions differ where |logit| >= 0.05"
    Hm = w.code.H.astype(np.int64)
    assert (syn.cpu().numpy() == (bits.cpu().numpy().astype(np.int64) @ Hm.T) % 2).all()
