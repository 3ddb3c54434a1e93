"""Python handle on the CPU oracle (oracle/aecct_oracle.c).  TEST INFRASTRUCTURE ONLY.

Only the tests, the smoke check and the CPU-baseline leg of the benchmark use this
module.  It compiles the plain C oracle with gcc (no fused multiply-add contraction,
no fast-math) and calls it through ctypes.  It never touches the CUDA library.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from typing import Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "aecct_oracle.c")
_OUT_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_OUT_DIR, "liboracle.so")
_lock = threading.Lock()
_lib = None

GCC_FLAGS = ["-O2", "-std=c11", "-fPIC", "-shared", "-fno-fast-math", "-ffp-contract=off", "-pthread"]


def build(force: bool = False) -> str:
    """Compile the oracle into oracle/_build/liboracle.so (skipped when up to date)."""
    os.makedirs(_OUT_DIR, exist_ok=True)
    if not force and os.path.exists(_LIB_PATH) and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    subprocess.check_call(["gcc", *GCC_FLAGS, _SRC, "-o", tmp, "-lm"])
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


class OracleModel(ctypes.Structure):
    _fields_ = [
        ("n", ctypes.c_int32), ("k", ctypes.c_int32), ("d", ctypes.c_int32), ("n_layers", ctypes.c_int32),
        ("heads", ctypes.c_int32), ("h_first", ctypes.c_int32), ("d_spe", ctypes.c_int32),
        ("ffn_mult", ctypes.c_int32), ("activation", ctypes.c_int32), ("mask_mode", ctypes.c_int32),
        ("alpha_mode", ctypes.c_int32), ("linear_mode", ctypes.c_int32),
        ("H", ctypes.c_void_p), ("emb", ctypes.c_void_p), ("spe", ctypes.c_void_p), ("w", ctypes.c_void_p),
        ("w_scale", ctypes.c_void_p), ("bias", ctypes.c_void_p), ("ln_gamma", ctypes.c_void_p),
        ("ln_beta", ctypes.c_void_p), ("w_d1", ctypes.c_void_p), ("b_d1", ctypes.c_float),
        ("w_out", ctypes.c_void_p), ("b_out", ctypes.c_void_p), ("ln_eps", ctypes.c_float),
        ("alpha_floor", ctypes.c_float), ("w_full", ctypes.c_void_p),
    ]


class OracleCapture(ctypes.Structure):
    _fields_ = [("cap_B", ctypes.c_int64), ("q", ctypes.c_void_p), ("acc", ctypes.c_void_p),
                ("alpha", ctypes.c_void_p), ("syn", ctypes.c_void_p)]


def lib():
    global _lib
    with _lock:
        if _lib is None:
            # AECCT_ORACLE_LIB names another build of this file (the planted-mistake tests run the
            # pins against copies of the oracle with one mistake each)
            path = os.environ.get("AECCT_ORACLE_LIB") or build()
            L = ctypes.CDLL(path)
            P = ctypes.c_void_p
            L.oracle_decode.argtypes = [ctypes.POINTER(OracleModel), P, ctypes.c_int64, P, P, P, ctypes.c_int,
                                        ctypes.POINTER(OracleCapture)]
            L.oracle_decode.restype = ctypes.c_int
            L.oracle_exp2_series.argtypes = [ctypes.c_float]
            L.oracle_exp2_series.restype = ctypes.c_float
            L.oracle_gelu.argtypes = [ctypes.c_float]
            L.oracle_gelu.restype = ctypes.c_float
            L.oracle_bf16_round.argtypes = [ctypes.c_float]
            L.oracle_bf16_round.restype = ctypes.c_float
            L.oracle_full_linear_row.argtypes = [P, ctypes.c_int, P, ctypes.c_int, P, P, P]
            L.oracle_psum.argtypes = [P, ctypes.c_int]
            L.oracle_psum.restype = ctypes.c_float
            L.oracle_hard_decision.argtypes = [P, ctypes.c_int, P]
            L.oracle_syndrome.argtypes = [P, ctypes.c_int, ctypes.c_int, P, P]
            L.oracle_masks.argtypes = [P, ctypes.c_int, ctypes.c_int, P, P]
            L.oracle_quant_row.argtypes = [P, ctypes.c_int, ctypes.c_float, P, P]
            L.oracle_aap_linear_row.argtypes = [P, ctypes.c_float, ctypes.c_int, P, ctypes.c_int, ctypes.c_float,
                                                P, P, P]
            L.oracle_ternary.argtypes = [P, ctypes.c_int64, ctypes.c_float, ctypes.c_float, P, P]
            L.oracle_ternary.restype = ctypes.c_int
            L.oracle_layernorm_row.argtypes = [P, ctypes.c_int, P, P, ctypes.c_float, P]
            L.oracle_attention.argtypes = [P, P, P, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int, P, P, P]
            L.oracle_exp2_coefficients.argtypes = [P]
            _lib = L
    return _lib


def _p(a: np.ndarray) -> int:
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data


# ---------------------------------------------------------------------------
# primitives (each a thin call into the C oracle)
# ---------------------------------------------------------------------------

def exp2_series(x) -> np.ndarray:
    L = lib()
    xs = np.asarray(x, dtype=np.float32).ravel()
    return np.array([L.oracle_exp2_series(float(v)) for v in xs], dtype=np.float32)


def gelu(x) -> np.ndarray:
    L = lib()
    xs = np.asarray(x, dtype=np.float32).ravel()
    return np.array([L.oracle_gelu(float(v)) for v in xs], dtype=np.float32)


def bf16_round(x) -> np.ndarray:
    L = lib()
    xs = np.asarray(x, dtype=np.float32).ravel()
    return np.array([L.oracle_bf16_round(float(v)) for v in xs], dtype=np.float32)


def full_linear_row(x, W, b):
    """The full-precision linear layer of one row: (fp32 sums before the bias, outputs)."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    W = np.ascontiguousarray(W, dtype=np.float32)
    b = np.ascontiguousarray(b, dtype=np.float32)
    N, K = W.shape
    s = np.zeros(N, np.float32)
    out = np.zeros(N, np.float32)
    lib().oracle_full_linear_row(_p(x), K, _p(W), N, _p(b), _p(s), _p(out))
    return s, out


def exp2_coefficients() -> np.ndarray:
    out = np.zeros(8, dtype=np.float32)
    lib().oracle_exp2_coefficients(_p(out))
    return out


def psum(v) -> np.float32:
    v = np.ascontiguousarray(v, dtype=np.float32)
    return np.float32(lib().oracle_psum(_p(v), v.size))


def hard_decision(y) -> np.ndarray:
    y = np.ascontiguousarray(y, dtype=np.float32)
    b = np.zeros(y.size, dtype=np.uint8)
    lib().oracle_hard_decision(_p(y), y.size, _p(b))
    return b


def syndrome(H, bits) -> np.ndarray:
    H = np.ascontiguousarray(H, dtype=np.uint8)
    b = np.ascontiguousarray(bits, dtype=np.uint8)
    s = np.zeros(H.shape[0], dtype=np.uint8)
    lib().oracle_syndrome(_p(H), H.shape[0], H.shape[1], _p(b), _p(s))
    return s


def masks(H):
    H = np.ascontiguousarray(H, dtype=np.uint8)
    m, n = H.shape
    T = n + m
    M1 = np.zeros((T, T), dtype=np.uint8)
    M2 = np.zeros((T, T), dtype=np.uint8)
    lib().oracle_masks(_p(H), m, n, _p(M1), _p(M2))
    return M1, M2


def quant_row(x, alpha_floor: float = 1e-5):
    x = np.ascontiguousarray(x, dtype=np.float32)
    q = np.zeros(x.size, dtype=np.int8)
    a = np.zeros(1, dtype=np.float32)
    lib().oracle_quant_row(_p(x), x.size, alpha_floor, _p(q), _p(a))
    return q, np.float32(a[0])


def aap_linear_row(q, alpha: float, W, s_w: float, b):
    q = np.ascontiguousarray(q, dtype=np.int8)
    W = np.ascontiguousarray(W, dtype=np.int8)
    b = np.ascontiguousarray(b, dtype=np.float32)
    N, K = W.shape
    acc = np.zeros(N, dtype=np.int32)
    out = np.zeros(N, dtype=np.float32)
    lib().oracle_aap_linear_row(_p(q), float(alpha), K, _p(W), N, float(s_w), _p(b), _p(acc), _p(out))
    return acc, out


def ternary(W, delta: float = 1.0, eps: float = 1e-8):
    W = np.ascontiguousarray(W, dtype=np.float32)
    t = np.zeros(W.shape, dtype=np.int8)
    sc = np.zeros(1, dtype=np.float32)
    rc = lib().oracle_ternary(_p(W), W.size, delta, eps, _p(t), _p(sc))
    assert rc == 0
    return t, np.float32(sc[0])


def layernorm_row(v, g, b, eps: float = 1e-5):
    v = np.ascontiguousarray(v, dtype=np.float32)
    g = np.ascontiguousarray(g, dtype=np.float32)
    b = np.ascontiguousarray(b, dtype=np.float32)
    y = np.zeros_like(v)
    lib().oracle_layernorm_row(_p(v), v.size, _p(g), _p(b), eps, _p(y))
    return y


def attention(Q, K, V, heads: int, h_first: int, M1, M2):
    Q = np.ascontiguousarray(Q, dtype=np.float32)
    K = np.ascontiguousarray(K, dtype=np.float32)
    V = np.ascontiguousarray(V, dtype=np.float32)
    M1 = np.ascontiguousarray(M1, dtype=np.uint8)
    M2 = np.ascontiguousarray(M2, dtype=np.uint8)
    T, d = Q.shape
    A = np.zeros_like(Q)
    lib().oracle_attention(_p(Q), _p(K), _p(V), T, d, heads, h_first, _p(M1), _p(M2), _p(A))
    return A


# ---------------------------------------------------------------------------
# whole decoder
# ---------------------------------------------------------------------------

class _Packed:
    """The model tensors laid out as the oracle's C struct expects (kept alive with it)."""

    def __init__(self, model):
        self.H = np.ascontiguousarray(model.H, dtype=np.uint8)
        self.emb = np.ascontiguousarray(model.emb, dtype=np.float32)
        self.spe = np.ascontiguousarray(model.spe, dtype=np.float32)
        self.w = np.ascontiguousarray(
            np.concatenate([np.asarray(t, dtype=np.int8).ravel() for layer in model.w_tern for t in layer])
            if model.n_layers else np.zeros(1, np.int8))
        self.w_scale = np.ascontiguousarray(model.w_scale, dtype=np.float32).reshape(-1)
        self.bias = np.ascontiguousarray(
            np.concatenate([np.asarray(b, dtype=np.float32).ravel() for layer in model.bias for b in layer])
            if model.n_layers else np.zeros(1, np.float32))
        self.ln_gamma = np.ascontiguousarray(model.ln_gamma, dtype=np.float32).reshape(-1)
        self.ln_beta = np.ascontiguousarray(model.ln_beta, dtype=np.float32).reshape(-1)
        self.w_d1 = np.ascontiguousarray(model.w_d1, dtype=np.float32)
        self.w_out = np.ascontiguousarray(model.w_out, dtype=np.float32)
        self.b_out = np.ascontiguousarray(model.b_out, dtype=np.float32)
        lm = int(getattr(model, "linear_mode", 0))
        self.w_full = (np.ascontiguousarray(np.concatenate(
            [np.asarray(w, np.float32).ravel() for layer in model.w_full for w in layer]))
            if lm == 1 else np.zeros(1, np.float32))
        if self.w_scale.size == 0:
            self.w_scale = np.zeros(1, np.float32)
            self.ln_gamma = np.zeros(1, np.float32)
            self.ln_beta = np.zeros(1, np.float32)
        self.st = OracleModel(
            model.n, model.k, model.d, model.n_layers, model.heads, model.h_first, model.d_spe, model.ffn_mult,
            model.activation, int(getattr(model, "mask_mode", 0)), int(getattr(model, "alpha_mode", 0)), lm,
            _p(self.H), _p(self.emb), _p(self.spe) if self.spe.size else None, _p(self.w),
            _p(self.w_scale), _p(self.bias), _p(self.ln_gamma), _p(self.ln_beta), _p(self.w_d1),
            float(model.b_d1), _p(self.w_out), _p(self.b_out), float(model.ln_eps), float(model.alpha_floor),
            _p(self.w_full) if lm == 1 else None)


def decode(model, y, nthreads: Optional[int] = None, cap_B: int = 0):
    """Run the oracle forward pass on y[B][n].

    Returns dict(bits uint8[B,n], syndrome uint8[B,n-k], logits float32[B,n]) and, when
    cap_B > 0, the integer-core record of the first cap_B codewords
    (q int8, acc int32, alpha float32, syn_in uint8) in the layout documented in the C file.
    """
    y = np.ascontiguousarray(y, dtype=np.float32)
    B, n = y.shape
    assert n == model.n
    m = model.n - model.k
    T = 2 * model.n - model.k
    pk = _Packed(model)
    bits = np.zeros((B, n), dtype=np.uint8)
    syn = np.zeros((B, m), dtype=np.uint8)
    logits = np.zeros((B, n), dtype=np.float32)
    cap = None
    capst = None
    if cap_B:
        cap_B = min(cap_B, B)
        W4 = 4 * model.d
        cap = dict(
            q=np.zeros((cap_B, model.n_layers, 4, T, W4), dtype=np.int8),
            acc=np.zeros((cap_B, model.n_layers, 4, T, W4), dtype=np.int32),
            alpha=np.zeros((cap_B, model.n_layers, 4, T), dtype=np.float32),
            syn_in=np.zeros((cap_B, m), dtype=np.uint8),
        )
        capst = OracleCapture(cap_B, _p(cap["q"]), _p(cap["acc"]), _p(cap["alpha"]), _p(cap["syn_in"]))
    if nthreads is None:
        nthreads = os.cpu_count() or 1
    rc = lib().oracle_decode(ctypes.byref(pk.st), _p(y), B, _p(bits), _p(syn), _p(logits), int(nthreads),
                             ctypes.byref(capst) if capst is not None else None)
    if rc != 0:
        raise ValueError(f"oracle_decode failed with status {rc}")
    out = dict(bits=bits, syndrome=syn, logits=logits)
    if cap is not None:
        out["capture"] = cap
    return out
