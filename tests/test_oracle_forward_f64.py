"""An independent float64 forward pass (numpy, written from the paper) against the oracle.

The integer core is teacher-forced: the oracle's recorded int32 accumulators of every GEMM
(exact: `test_capture_integer_core_consistent` checks them against q . W) feed the float64
pass, which recomputes everything in between on its own -- embedding with the syndrome tokens
(Sec. 3), dequantisation (eq. AAPLinear), masked multi-head softmax attention with masks built
here from H (Sec. 4.2, or the ECCT code-aware mask of Sec. 3 when mask_mode = 1), residual +
LayerNorm (Post-LN, Sec. 5), ReLU (or GELU) FFN, the output head -- and checks at every quantised GEMM
input that the oracle's alpha is max|x| and its int8 codes are rint(x * 127 / alpha) of this
float64 x, and finally that the logits agree.  A dropped term, a wrong index, a transposed
operand or a mask mistake in the oracle changes codes or logits far beyond fp32 rounding.
"""
import math

import numpy as np
import pytest

from f64_forward import forward64, ln64, masks64
from oracle import oracle as O
from paper_2410_05911_gb300 import inputs as I


@pytest.mark.parametrize("key,d,layers,var", [
    ("hamming7_4", 32, 2, dict()),
    ("bch31_16", 32, 2, dict()),
    ("bch31_16", 32, 2, dict(h_first=2)),
    ("bch31_16", 32, 2, dict(mask_mode=1)),
    ("polar64_32", 64, 1, dict(mask_mode=1, binary=True)),
    ("bch31_16", 32, 2, dict(alpha_mode=1)),
    ("polar64_32", 64, 1, dict(alpha_mode=1, h_first=6)),
    ("bch31_16", 32, 2, dict(activation=1)),
    ("polar64_32", 64, 1, dict(activation=1, mask_mode=1)),
])
def test_oracle_matches_float64_forward(key, d, layers, var):
    code = I.make_code(key)
    var = dict(var)
    mask_mode = var.pop("mask_mode", 0)
    alpha_mode = var.pop("alpha_mode", 0)
    model = I.random_model(code, d, layers, seed=41, **var)
    model.mask_mode = mask_mode
    model.alpha_mode = alpha_mode
    B = 3
    y = I.channel_batch(code, B, 2.0, seed=43).y
    r = O.decode(model, y, nthreads=2, cap_B=B)
    logits, boundary = forward64(model, y, r["capture"])
    assert boundary <= 2  # codes exactly at a rounding boundary are rare
    assert np.abs(r["logits"] - logits).max() < 1e-3 * (1.0 + np.abs(logits).max())


def test_casa_mask_is_independent_of_head_split():
    # with the ECCT mask every head sees the same keys, so h_first cannot matter
    code = I.make_code("bch31_16")
    y = I.channel_batch(code, 4, 2.0, seed=5).y
    outs = []
    for hf in (0, 3, 8):
        model = I.random_model(code, 32, 2, seed=7, h_first=hf)
        model.mask_mode = 1
        outs.append(O.decode(model, y, nthreads=2)["logits"])
    assert all((o.view(np.int32) == outs[0].view(np.int32)).all() for o in outs)


def _bf16(a):
    # round to nearest even to bf16 with torch's conversion (independent of the oracle's own)
    torch = pytest.importorskip("torch")
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(torch.bfloat16).to(torch.float64).numpy()


def forward64_full(model, y):
    """Float64 forward pass with full-precision linear layers (ECCT, Sec. 3): every linear input
    and weight rounded to bf16, everything else in float64."""
    H = model.H
    m, n = H.shape
    T, d, heads = n + m, model.d, model.heads
    dh = d // heads
    M1, M2 = masks64(H, model.mask_mode)
    logits = np.zeros((y.shape[0], n))
    lin = lambda x, W, b: _bf16(x) @ _bf16(W).T + b.astype(np.float64)  # noqa: E731
    for bi in range(y.shape[0]):
        yb = y[bi].astype(np.float64)
        s = (H.astype(np.int64) @ (yb < 0).astype(np.int64)) % 2
        h = np.concatenate([np.abs(yb), 1.0 - 2.0 * s])
        # the embedding product is one fp32 multiply in every implementation
        x = np.concatenate([(h.astype(np.float32)[:, None] * model.emb).astype(np.float64),
                            model.spe.astype(np.float64)], 1)
        for l in range(model.n_layers):
            Wq, Wk, Wv, Wo, W1, W2 = model.w_full[l]
            bq, bk, bv, bo, b1, b2 = model.bias[l]
            Q, K, V = lin(x, Wq, bq), lin(x, Wk, bk), lin(x, Wv, bv)
            A = np.zeros((T, d))
            for e in range(heads):
                M = M1 if e < model.h_first else M2
                sl = slice(e * dh, (e + 1) * dh)
                S = np.where(M, Q[:, sl] @ K[:, sl].T / np.sqrt(dh), -np.inf)
                P = np.exp(S - S.max(1, keepdims=True))
                A[:, sl] = (P / P.sum(1, keepdims=True)) @ V[:, sl]
            x = ln64(x + lin(A, Wo, bo), model.ln_gamma[l, 0], model.ln_beta[l, 0], model.ln_eps)
            u = lin(x, W1, b1)
            if model.activation == 0:
                u = np.maximum(u, 0.0)
            else:
                u = 0.5 * u * (1.0 + np.vectorize(math.erf)(u / math.sqrt(2.0)))
            x = ln64(x + lin(u, W2, b2), model.ln_gamma[l, 1], model.ln_beta[l, 1], model.ln_eps)
        z = x @ model.w_d1.astype(np.float64) + model.b_d1
        logits[bi] = z @ model.w_out.astype(np.float64) + model.b_out
    return logits


@pytest.mark.parametrize("key,d,layers,var", [
    ("bch31_16", 32, 2, dict()),
    ("polar64_32", 64, 2, dict(activation=1)),
    ("bch31_16", 32, 2, dict(activation=1, mask_mode=1)),  # the ECCT configuration
])
def test_oracle_full_precision_matches_float64_forward(key, d, layers, var):
    # not teacher-forced: the fp32 rounding between the float64 pass and the oracle can move a
    # bf16 rounding of a linear input by one bf16 step (2^-8 relative) now and then, so the
    # logits agree to about 1e-3 rather than to fp32 rounding
    code = I.make_code(key)
    var = dict(var)
    mask_mode = var.pop("mask_mode", 0)
    model = I.random_model(code, d, layers, seed=21, full_precision=True, **var)
    model.mask_mode = mask_mode
    y = I.channel_batch(code, 3, 2.0, seed=23).y
    r = O.decode(model, y, nthreads=2)
    ref = forward64_full(model, y)
    assert np.abs(r["logits"] - ref).max() < 2e-2 * (1.0 + np.abs(ref).max())
    assert np.median(np.abs(r["logits"] - ref)) < 1e-4 * (1.0 + np.abs(ref).max())
