"""An independent float64 forward pass of the AECCT decoder (numpy, written from the paper),
teacher-forced on a recorded integer core.

Given the int8 codes, alpha and int32 accumulators that one implementation recorded for every
GEMM of a word (eq. Quant, eq. AAPLinear of Sec. 4.1), it recomputes everything in between on
its own in float64: the embedding with the syndrome tokens (Sec. 3), dequantisation, masked
multi-head softmax attention with masks built here from H (Sec. 4.2, or the ECCT code-aware
mask of Sec. 3 when mask_mode = 1), residual + LayerNorm (Post-LN, Sec. 5), the ReLU (or GELU)
feed-forward layer and the output head.  At every quantised GEMM input it checks that the
recorded alpha is max|x| of this float64 x and that the recorded codes are rint(x * 127 / alpha)
except at a rounding boundary.  It shares nothing with the oracle or the CUDA path.
"""
import math

import numpy as np


def masks64(H, mask_mode):
    m, n = H.shape
    T = n + m
    Hi = H.astype(np.int64)
    M1 = np.zeros((T, T), bool)
    M1[:n, n:] = Hi.T > 0
    M1[n:, :n] = Hi > 0
    M2 = np.zeros((T, T), bool)
    M2[:n, :n] = (Hi.T @ Hi) > 0
    M2[n:, n:] = (Hi @ Hi.T) > 0
    if mask_mode == 1:
        M1 = M2 = M1 | M2
    return M1, M2


def ln64(v, g, b, eps):
    mu = v.mean(-1, keepdims=True)
    var = ((v - mu) ** 2).mean(-1, keepdims=True)
    return (v - mu) / np.sqrt(var + eps) * g + b


def check_quant(x, q, alpha, floor, label, per_word=False):
    # per token (C-1): alpha_t = max(max_i |x_ti|, floor); per word: one max over the matrix
    a = np.maximum(np.abs(x).max(1), floor)
    if per_word:
        a = np.full_like(a, a.max())
    assert (np.abs(alpha - a) <= 1e-5 * a).all(), f"{label}: alpha {alpha} vs {a}"
    v = x * (127.0 / a)[:, None]
    ref = np.rint(v)
    bad = q.astype(np.int64) != ref
    # a code may differ from the float64 rounding only at a rounding boundary
    near = np.abs(np.abs(v - np.floor(v)) - 0.5) < 1e-3
    assert not (bad & ~near).any(), f"{label}: {int((bad & ~near).sum())} codes differ away from a boundary"
    return int(bad.sum())


def forward64(model, y, cap):
    H = model.H
    m, n = H.shape
    T, d, heads = n + m, model.d, model.heads
    dh = d // heads
    F = model.ffn_mult * d
    M1, M2 = masks64(H, model.mask_mode)
    q, acc, alpha = cap["q"], cap["acc"], cap["alpha"]
    pw = getattr(model, "alpha_mode", 0) == 1
    boundary = 0
    logits = np.zeros((y.shape[0], n))
    for b in range(q.shape[0]):
        yb = y[b].astype(np.float64)
        s = (H.astype(np.int64) @ (yb < 0).astype(np.int64)) % 2
        h = np.concatenate([np.abs(yb), 1.0 - 2.0 * s])
        x = np.concatenate([h[:, None] * model.emb.astype(np.float64), model.spe.astype(np.float64)], 1)
        for l in range(model.n_layers):
            sw = model.w_scale[l].astype(np.float64)
            bias = [bb.astype(np.float64) for bb in model.bias[l]]
            # QKV
            boundary += check_quant(x, q[b, l, 0, :, :d], alpha[b, l, 0], model.alpha_floor, f"b{b} l{l} qkv", pw)
            f = alpha[b, l, 0][:, None] / 127.0
            A0 = acc[b, l, 0, :, :3 * d].astype(np.float64)
            Q = A0[:, :d] * (sw[0] * f) + bias[0]
            K = A0[:, d:2 * d] * (sw[1] * f) + bias[1]
            V = A0[:, 2 * d:] * (sw[2] * f) + bias[2]
            # attention: heads [0, h_first) on M1, the rest on M2, scale 1/sqrt(d_h)
            A = np.zeros((T, d))
            for e in range(heads):
                M = M1 if e < model.h_first else M2
                sl = slice(e * dh, (e + 1) * dh)
                S = Q[:, sl] @ K[:, sl].T / np.sqrt(dh)
                S = np.where(M, S, -np.inf)
                P = np.exp(S - S.max(1, keepdims=True))
                P /= P.sum(1, keepdims=True)
                A[:, sl] = P @ V[:, sl]
            # O projection, residual, LayerNorm
            boundary += check_quant(A, q[b, l, 1, :, :d], alpha[b, l, 1], model.alpha_floor, f"b{b} l{l} o", pw)
            o = acc[b, l, 1, :, :d].astype(np.float64) * (sw[3] * alpha[b, l, 1][:, None] / 127.0) + bias[3]
            x = ln64(x + o, model.ln_gamma[l, 0], model.ln_beta[l, 0], model.ln_eps)
            # FFN
            boundary += check_quant(x, q[b, l, 2, :, :d], alpha[b, l, 2], model.alpha_floor, f"b{b} l{l} ffn1", pw)
            u = acc[b, l, 2, :, :F].astype(np.float64) * (sw[4] * alpha[b, l, 2][:, None] / 127.0) + bias[4]
            if model.activation == 0:
                u = np.maximum(u, 0.0)
            else:  # GELU(u) = u Phi(u) with the exact erf
                u = 0.5 * u * (1.0 + np.vectorize(math.erf)(u / math.sqrt(2.0)))
            boundary += check_quant(u, q[b, l, 3, :, :F], alpha[b, l, 3], model.alpha_floor, f"b{b} l{l} ffn2", pw)
            o2 = acc[b, l, 3, :, :d].astype(np.float64) * (sw[5] * alpha[b, l, 3][:, None] / 127.0) + bias[5]
            x = ln64(x + o2, model.ln_gamma[l, 1], model.ln_beta[l, 1], model.ln_eps)
        z = x @ model.w_d1.astype(np.float64) + model.b_d1
        logits[b] = z @ model.w_out.astype(np.float64) + model.b_out
    return logits, boundary
