"""Python handle on the SPE oracle (oracle/spe_oracle.c).  TEST INFRASTRUCTURE ONLY.

Only the tests use this module.  It compiles the plain C restatement of the spectral positional
encoding (Sec. 4.3: Tanner-graph Laplacian, cyclic Jacobi eigensolver, canonical eigenbasis,
multi-head self-attention over the eigen-tokens, average pooling) with gcc and calls it through
ctypes.  It never touches the CUDA library or the package's host precompute.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "spe_oracle.c")
_OUT_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_OUT_DIR, "libspe_oracle.so")
_lock = threading.Lock()
_lib = None

CLUSTER_TOL = 1e-8
VANISH_TOL = 1e-6


def build(force: bool = False) -> str:
    os.makedirs(_OUT_DIR, exist_ok=True)
    if not force and os.path.exists(_LIB_PATH) and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    subprocess.check_call(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fno-fast-math", _SRC, "-o", tmp, "-lm"])
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def lib():
    global _lib
    with _lock:
        if _lib is None:
            L = ctypes.CDLL(build())
            P, I, D = ctypes.c_void_p, ctypes.c_int, ctypes.c_double
            L.spe_oracle_laplacian.argtypes = [P, I, I, P]
            L.spe_oracle_jacobi.argtypes = [P, I, P, P]
            L.spe_oracle_jacobi.restype = I
            L.spe_oracle_canonical.argtypes = [P, P, I, D, D]
            L.spe_oracle_canonical.restype = I
            L.spe_oracle_mhsa.argtypes = [P, P, I, P, I, I, I, P, P, P, P, P, P]
            L.spe_oracle_table.argtypes = [P, I, I, I, I, P, P, P, P, P, D, D, P, I, P, P, P]
            L.spe_oracle_table.restype = I
            _lib = L
    return _lib


def _c(a, dtype=np.float64):
    return np.ascontiguousarray(a, dtype=dtype)


def laplacian(H) -> np.ndarray:
    H = _c(H, np.uint8)
    m, n = H.shape
    L = np.zeros((n + m, n + m))
    lib().spe_oracle_laplacian(H.ctypes.data, n, m, L.ctypes.data)
    return L


def jacobi(S):
    """Eigenvalues (unsorted) and eigenvectors (columns) of a symmetric matrix, and the sweeps."""
    S = _c(S).copy()
    T = S.shape[0]
    lam, V = np.zeros(T), np.zeros((T, T))
    sweeps = lib().spe_oracle_jacobi(S.ctypes.data, T, lam.ctypes.data, V.ctypes.data)
    return lam, V, sweeps


def canonical(lam, V, cluster_tol: float = CLUSTER_TOL, vanish_tol: float = VANISH_TOL):
    lam, V = _c(lam).copy(), _c(V).copy()
    rc = lib().spe_oracle_canonical(lam.ctypes.data, V.ctypes.data, lam.shape[0], cluster_tol, vanish_tol)
    if rc != 0:
        raise ValueError("canonical eigenbasis failed")
    return lam, V


def mhsa(lam, V, p, nodes=None) -> np.ndarray:
    lam, V = _c(lam), _c(V)
    T = lam.shape[0]
    nodes = _c(np.arange(T) if nodes is None else nodes, np.int32)
    heads, d_spe = p.wq.shape[0], p.w_pe.shape[1]
    out = np.zeros((nodes.shape[0], d_spe))
    ws = [_c(p.w_pe), _c(p.wq), _c(p.wk), _c(p.wv), _c(p.wo)]
    lib().spe_oracle_mhsa(lam.ctypes.data, V.ctypes.data, T, nodes.ctypes.data, nodes.shape[0], d_spe, heads,
                          *[w.ctypes.data for w in ws], out.ctypes.data)
    return out


def table(H, p, nodes=None):
    """(SPE rows of `nodes` (all by default) [nn, d_spe], canonical eigenvalues, eigenvectors)."""
    H = _c(H, np.uint8)
    m, n = H.shape
    T = n + m
    nodes = _c(np.arange(T) if nodes is None else nodes, np.int32)
    heads, d_spe = p.wq.shape[0], p.w_pe.shape[1]
    lam, V = np.zeros(T), np.zeros((T, T))
    out = np.zeros((nodes.shape[0], d_spe))
    ws = [_c(p.w_pe), _c(p.wq), _c(p.wk), _c(p.wv), _c(p.wo)]
    rc = lib().spe_oracle_table(H.ctypes.data, n, m, d_spe, heads, *[w.ctypes.data for w in ws], CLUSTER_TOL,
                                VANISH_TOL, nodes.ctypes.data, nodes.shape[0], lam.ctypes.data, V.ctypes.data,
                                out.ctypes.data)
    if rc < 0:
        raise ValueError("SPE oracle: canonical eigenbasis failed")
    return out, lam, V
