"""Python binding of libaecct (the C ABI in include/aecct.h).

Argument marshalling only: every step of the decoder runs in the CUDA library.  PyTorch
provides device memory and streams.  There is no CPU fallback: if the library cannot be
loaded, or no sm_103 GPU is present, the calls raise.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Tuple

import numpy as np

from . import build_lib

AECCT_OK = 0
AECCT_ERR_INVALID_ARG = -1
AECCT_ERR_UNSUPPORTED = -2
AECCT_ERR_OUT_OF_MEMORY = -3
AECCT_ERR_CUDA = -4
AECCT_ERR_TIMEOUT = -5
AECCT_ERR_NO_DEVICE = -6

EXPORTED_SYMBOLS = (
    "aecct_create", "aecct_decode", "aecct_decode_host", "aecct_synchronize", "aecct_set_capture",
    "aecct_query", "aecct_destroy", "aecct_status_string", "aecct_last_error", "aecct_selftest_mma",
    "aecct_selftest_timeout", "aecct_decode_host_noalloc", "aecct_selftest_fma_rate", "aecct_aap_ternarize",
    "aecct_spe_table",
)


class AecctError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        super().__init__(f"{what}: {status_string(status)} ({status}) {last_error()}".strip())


class ModelDesc(ctypes.Structure):
    _fields_ = [
        ("n", ctypes.c_int32), ("k", ctypes.c_int32), ("d", ctypes.c_int32), ("n_layers", ctypes.c_int32),
        ("heads", ctypes.c_int32), ("h_first", ctypes.c_int32), ("d_spe", ctypes.c_int32),
        ("ffn_mult", ctypes.c_int32), ("activation", ctypes.c_int32), ("cluster_ctas", ctypes.c_int32),
        ("attention_mode", ctypes.c_int32), ("mask_mode", ctypes.c_int32),
        ("alpha_mode", ctypes.c_int32), ("linear_mode", ctypes.c_int32),
        ("H", ctypes.c_void_p), ("emb", ctypes.c_void_p), ("spe", ctypes.c_void_p), ("w_packed", ctypes.c_void_p),
        ("w_scale", ctypes.c_void_p), ("bias", ctypes.c_void_p), ("ln_gamma", ctypes.c_void_p),
        ("ln_beta", ctypes.c_void_p), ("w_d1", ctypes.c_void_p), ("b_d1", ctypes.c_float),
        ("w_out", ctypes.c_void_p), ("b_out", ctypes.c_void_p), ("ln_eps", ctypes.c_float),
        ("alpha_floor", ctypes.c_float), ("wait_limit_cycles", ctypes.c_int64), ("w_full", ctypes.c_void_p),
    ]


_lib = None


def library_path() -> str:
    return build_lib.LIB_PATH


def load(build_if_missing: bool = True):
    """Load libaecct.so from the package's _build directory (building it if asked)."""
    global _lib
    if _lib is not None:
        return _lib
    path = build_lib.LIB_PATH
    if not os.path.exists(path):
        if not build_if_missing:
            raise OSError(f"libaecct.so not built at {path}")
        build_lib.build()
    L = ctypes.CDLL(path)
    P, I32, I64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
    L.aecct_create.argtypes = [ctypes.POINTER(ModelDesc), ctypes.POINTER(P)]
    L.aecct_decode.argtypes = [P, P, I64, P, P, P, P]
    L.aecct_decode_host.argtypes = [P, P, I64, P, P, P, P]
    L.aecct_decode_host_noalloc.argtypes = [P, P, I64, P, P, P, P]
    L.aecct_synchronize.argtypes = [P]
    L.aecct_set_capture.argtypes = [P, I64, P, P, P, P]
    L.aecct_query.argtypes = [P] + [ctypes.POINTER(I32)] * 6
    L.aecct_destroy.argtypes = [P]
    L.aecct_status_string.argtypes = [ctypes.c_int]
    L.aecct_status_string.restype = ctypes.c_char_p
    L.aecct_last_error.argtypes = []
    L.aecct_last_error.restype = ctypes.c_char_p
    L.aecct_selftest_mma.argtypes = [P, P, I32, I32, P]
    L.aecct_selftest_timeout.argtypes = [I64, ctypes.POINTER(I32)]
    L.aecct_selftest_fma_rate.argtypes = [I32, ctypes.POINTER(ctypes.c_double)]
    L.aecct_aap_ternarize.argtypes = [P, I32, P, P, ctypes.c_float, P, P, P, P]
    L.aecct_spe_table.argtypes = [P, I32, I32, I32, I32, P, P, P, P, P, P, P, P, P]
    for name in EXPORTED_SYMBOLS:
        fn = getattr(L, name)
        if fn.restype is None or fn.restype is ctypes.c_int:
            if name not in ("aecct_status_string", "aecct_last_error"):
                fn.restype = ctypes.c_int
    _lib = L
    return L


def status_string(status: int) -> str:
    return load().aecct_status_string(int(status)).decode()


def last_error() -> str:
    return load().aecct_last_error().decode()


def _check(status: int, what: str) -> None:
    if status != AECCT_OK:
        raise AecctError(status, what)


def pack_ternary(t: np.ndarray) -> np.ndarray:
    """Pack int8 ternary values [rows][cols] (cols % 4 == 0) into the 2-bit ABI format:
    value i of a row goes to bits 2*(i%4) of byte i/4, coded 0 -> 00, +1 -> 01, -1 -> 11."""
    t = np.asarray(t, dtype=np.int8)
    rows, cols = t.shape
    assert cols % 4 == 0
    code = np.where(t == 1, 1, np.where(t == -1, 3, 0)).astype(np.uint8)
    if not np.isin(t, (-1, 0, 1)).all():
        raise ValueError("ternary weights must be in {-1, 0, 1}")
    c = code.reshape(rows, cols // 4, 4)
    return (c[..., 0] | (c[..., 1] << 2) | (c[..., 2] << 4) | (c[..., 3] << 6)).astype(np.uint8)


class _HostModel:
    """Contiguous host copies of a model's tensors, in the ABI layout (kept alive with the desc)."""

    def __init__(self, model, cluster_ctas: int = 0, wait_limit_cycles: int = 0, attention_mode: int = 0):
        d, F = model.d, model.ffn_mult * model.d
        self.H = np.ascontiguousarray(model.H, dtype=np.uint8)
        self.emb = np.ascontiguousarray(model.emb, dtype=np.float32)
        self.spe = np.ascontiguousarray(model.spe, dtype=np.float32)
        linear_mode = int(getattr(model, "linear_mode", 0))
        # AAP linears: 2-bit ternary codes and scales; full-precision linears (linear_mode 1): fp32
        # weights in the same per-block order (the arrays the mode does not read stay NULL)
        w_full = getattr(model, "w_full", None)
        if linear_mode != 1:
            packed = [pack_ternary(t).ravel() for layer in model.w_tern for t in layer]
            self.w_packed = np.ascontiguousarray(np.concatenate(packed) if packed else np.zeros(1, np.uint8))
            self.w_scale = np.ascontiguousarray(model.w_scale, dtype=np.float32).reshape(-1)
        else:
            self.w_packed = np.zeros(0, np.uint8)
            self.w_scale = np.zeros(0, np.float32)
        self.w_full = (np.ascontiguousarray(np.concatenate([np.asarray(w, np.float32).ravel()
                                                            for layer in w_full for w in layer]))
                       if linear_mode != 0 and w_full is not None else np.zeros(0, np.float32))
        self.bias = np.ascontiguousarray(
            np.concatenate([np.asarray(b, np.float32).ravel() for layer in model.bias for b in layer]))
        self.ln_gamma = np.ascontiguousarray(model.ln_gamma, dtype=np.float32).reshape(-1)
        self.ln_beta = np.ascontiguousarray(model.ln_beta, dtype=np.float32).reshape(-1)
        self.w_d1 = np.ascontiguousarray(model.w_d1, dtype=np.float32)
        self.w_out = np.ascontiguousarray(model.w_out, dtype=np.float32)
        self.b_out = np.ascontiguousarray(model.b_out, dtype=np.float32)
        ptr = lambda a: a.ctypes.data if a.size else None  # noqa: E731
        self.desc = ModelDesc(
            model.n, model.k, model.d, model.n_layers, model.heads, model.h_first, model.d_spe, model.ffn_mult,
            model.activation, int(cluster_ctas), int(attention_mode), int(getattr(model, "mask_mode", 0)),
            int(getattr(model, "alpha_mode", 0)), linear_mode, ptr(self.H), ptr(self.emb), ptr(self.spe),
            ptr(self.w_packed), ptr(self.w_scale), ptr(self.bias), ptr(self.ln_gamma), ptr(self.ln_beta),
            ptr(self.w_d1), float(model.b_d1), ptr(self.w_out), ptr(self.b_out), float(model.ln_eps),
            float(model.alpha_floor), int(wait_limit_cycles), ptr(self.w_full))


def create_handle(model, cluster_ctas: int = 0, wait_limit_cycles: int = 0, attention_mode: int = 0):
    """aecct_create on a model (see inputs.ModelTensors); returns (status, handle or None)."""
    L = load()
    hm = _HostModel(model, cluster_ctas, wait_limit_cycles, attention_mode)
    h = ctypes.c_void_p()
    st = L.aecct_create(ctypes.byref(hm.desc), ctypes.byref(h))
    return st, (h if st == AECCT_OK else None)


def check_outputs(out, B: int, n: int, m: int, device):
    """Caller-provided decode outputs (bits, syndrome or None, logits or None).  The kernel writes
    B full rows of each, so their shapes, types and device are checked here: the C ABI sees only
    pointers."""
    import torch

    bits, syn, logits = out
    for name, t, shape, dtype, required in (("bits", bits, (B, n), torch.uint8, True),
                                            ("syndrome", syn, (B, m), torch.uint8, False),
                                            ("logits", logits, (B, n), torch.float32, False)):
        if t is None and not required:
            continue
        if t is None or t.device != device or t.dtype != dtype or tuple(t.shape) != shape or not t.is_contiguous():
            raise ValueError(f"out {name} must be a contiguous {dtype} tensor of shape {shape} on {device}")
    return bits, syn, logits


class Decoder:
    """A decoder handle on the current CUDA device.

    decode(y) takes a float32 CUDA tensor [B, n] and returns (bits uint8 [B, n],
    syndrome uint8 [B, n-k] or None, logits float32 [B, n] or None), computed on
    torch.cuda.current_stream().
    """

    def __init__(self, model, cluster_ctas: int = 0, wait_limit_cycles: int = 0, attention_mode: int = 0):
        import torch

        if not torch.cuda.is_available():
            raise AecctError(AECCT_ERR_NO_DEVICE, "Decoder")
        self._torch = torch
        self.n, self.k = model.n, model.k
        self.m = model.n - model.k
        self.T = 2 * model.n - model.k
        self.d, self.n_layers = model.d, model.n_layers
        self._L = load()
        st, h = create_handle(model, cluster_ctas, wait_limit_cycles, attention_mode)
        _check(st, "aecct_create")
        self._h = h
        self._cap = None

    def close(self) -> None:
        if getattr(self, "_h", None) is not None:
            self._L.aecct_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def query(self) -> dict:
        vals = [ctypes.c_int32() for _ in range(6)]
        _check(self._L.aecct_query(self._h, *[ctypes.byref(v) for v in vals]), "aecct_query")
        keys = ("cluster_ctas", "words_per_group", "max_clusters", "threads_per_cta", "smem_bytes", "attention_mode")
        return {k: v.value for k, v in zip(keys, vals)}

    def decode(self, y, want_syndrome: bool = True, want_logits: bool = True, out=None, stream=None):
        torch = self._torch
        if not (y.is_cuda and y.dtype == torch.float32 and y.dim() == 2 and y.shape[1] == self.n):
            raise ValueError("y must be a float32 CUDA tensor of shape [B, n]")
        y = y.contiguous()
        B = y.shape[0]
        if out is None:
            bits = torch.empty((B, self.n), dtype=torch.uint8, device=y.device)
            syn = torch.empty((B, self.m), dtype=torch.uint8, device=y.device) if want_syndrome else None
            logits = torch.empty((B, self.n), dtype=torch.float32, device=y.device) if want_logits else None
        else:
            bits, syn, logits = check_outputs(out, B, self.n, self.m, y.device)
        s = stream if stream is not None else torch.cuda.current_stream(y.device)
        st = self._L.aecct_decode(self._h, y.data_ptr(), B, bits.data_ptr(), syn.data_ptr() if syn is not None else None,
                                  logits.data_ptr() if logits is not None else None, s.cuda_stream)
        _check(st, "aecct_decode")
        return bits, syn, logits

    def decode_host(self, y: np.ndarray, want_syndrome: bool = True, want_logits: bool = True):
        """End-to-end call with host arrays: copies in, decodes, copies out, waits."""
        y = self._host_y(y)
        B = y.shape[0]
        bits = np.empty((B, self.n), np.uint8)
        syn = np.empty((B, self.m), np.uint8) if want_syndrome else None
        logits = np.empty((B, self.n), np.float32) if want_logits else None
        st = self._L.aecct_decode_host(self._h, y.ctypes.data, B, bits.ctypes.data,
                                       syn.ctypes.data if syn is not None else None,
                                       logits.ctypes.data if logits is not None else None, None)
        _check(st, "aecct_decode_host")
        return bits, syn, logits

    def decode_host_noalloc(self, y: np.ndarray, want_syndrome: bool = True, want_logits: bool = True):
        """aecct_decode_host_noalloc: host arrays, device staging from the library's static scratch
        (no allocation).  Returns (status, bits, syndrome, logits); calls must not overlap."""
        y = self._host_y(y)
        B = y.shape[0]
        bits = np.empty((B, self.n), np.uint8)
        syn = np.empty((B, self.m), np.uint8) if want_syndrome else None
        logits = np.empty((B, self.n), np.float32) if want_logits else None
        st = self._L.aecct_decode_host_noalloc(self._h, y.ctypes.data, B, bits.ctypes.data,
                                               syn.ctypes.data if syn is not None else None,
                                               logits.ctypes.data if logits is not None else None, None)
        return st, bits, syn, logits

    def _host_y(self, y) -> np.ndarray:
        y = np.ascontiguousarray(y, dtype=np.float32)
        if y.ndim != 2 or y.shape[1] != self.n:
            raise ValueError(f"y must be a float32 array of shape [B, {self.n}]")
        return y

    def synchronize(self) -> int:
        return self._L.aecct_synchronize(self._h)

    def set_capture(self, cap_B: int):
        """Allocate capture buffers for the first cap_B words (0 disables); returns the tensors."""
        torch = self._torch
        if cap_B <= 0:
            _check(self._L.aecct_set_capture(self._h, 0, None, None, None, None), "aecct_set_capture")
            self._cap = None
            return None
        W = 4 * self.d
        dev = torch.device("cuda", torch.cuda.current_device())
        cap = dict(
            q=torch.zeros((cap_B, self.n_layers, 4, self.T, W), dtype=torch.int8, device=dev),
            acc=torch.zeros((cap_B, self.n_layers, 4, self.T, W), dtype=torch.int32, device=dev),
            alpha=torch.zeros((cap_B, self.n_layers, 4, self.T), dtype=torch.float32, device=dev),
            syn_in=torch.zeros((cap_B, self.m), dtype=torch.uint8, device=dev),
        )
        _check(self._L.aecct_set_capture(self._h, cap_B, cap["q"].data_ptr(), cap["acc"].data_ptr(),
                                         cap["alpha"].data_ptr(), cap["syn_in"].data_ptr()), "aecct_set_capture")
        self._cap = cap
        return cap


def selftest_mma(a: np.ndarray, b: np.ndarray) -> np.ndarray:
    """tcgen05 MMA self-test: returns A [128, K] @ B[N, K]^T computed on the tensor cores."""
    a = np.ascontiguousarray(a, dtype=np.int8)
    b = np.ascontiguousarray(b, dtype=np.int8)
    assert a.shape[0] == 128 and a.shape[1] == b.shape[1]
    out = np.zeros((128, b.shape[0]), np.float32)
    _check(load().aecct_selftest_mma(a.ctypes.data, b.ctypes.data, a.shape[1], b.shape[0], out.ctypes.data),
           "aecct_selftest_mma")
    return out


def selftest_timeout(limit_cycles: int) -> int:
    st = ctypes.c_int32(99)
    _check(load().aecct_selftest_timeout(int(limit_cycles), ctypes.byref(st)), "aecct_selftest_timeout")
    return st.value


def selftest_fma_rate(paired: bool) -> float:
    """Measured fp32 FMAs per second of the current device (scalar or paired f32x2 instructions)."""
    v = ctypes.c_double()
    _check(load().aecct_selftest_fma_rate(1 if paired else 0, ctypes.byref(v)), "aecct_selftest_fma_rate")
    return v.value


def aap_ternarize(tensors, delta=None, eps: float = 1e-8, want_weights: bool = False, stream=None):
    """aecct_aap_ternarize: eq. Ternary on the GPU for a list of float32 CUDA tensors (each with a
    multiple of 4 elements).  Returns (packed uint8 codes per tensor, scales float32 [n], and the
    weights scale * Ternary(W) per tensor when want_weights)."""
    import torch

    if not tensors:
        return [], None, None
    dev = tensors[0].device
    flat = torch.cat([t.reshape(-1).to(torch.float32) for t in tensors]).contiguous()
    lens = np.array([t.numel() for t in tensors], np.int64)
    deltas = np.asarray(delta if delta is not None else np.ones(len(tensors)), np.float32)
    packed = torch.empty(int(lens.sum()) // 4, dtype=torch.uint8, device=dev)
    scale = torch.empty(len(tensors), dtype=torch.float32, device=dev)
    wq = torch.empty_like(flat) if want_weights else None
    s = stream if stream is not None else torch.cuda.current_stream(dev)
    _check(load().aecct_aap_ternarize(flat.data_ptr(), len(tensors), lens.ctypes.data, deltas.ctypes.data, float(eps),
                                      packed.data_ptr(), scale.data_ptr(), wq.data_ptr() if wq is not None else None,
                                      s.cuda_stream), "aecct_aap_ternarize")
    offs = np.concatenate([[0], np.cumsum(lens)])
    codes = [packed[offs[j] // 4:offs[j + 1] // 4] for j in range(len(tensors))]
    wqs = [wq[offs[j]:offs[j + 1]].view(tensors[j].shape) for j in range(len(tensors))] if wq is not None else None
    return codes, scale, wqs


def spe_table(H: np.ndarray, params, want_eigen: bool = False):
    """aecct_spe_table: the SPE table of Sec. 4.3 computed on the GPU for parity-check matrix H and the
    SPE parameters (w_pe, wq, wk, wv, wo).  Returns the fp32 table [T, d_spe], and with want_eigen
    also (the fp64 table, eigenvalues [T], canonical eigenvectors [T, T])."""
    H = np.ascontiguousarray(H, np.uint8)
    m, n = H.shape
    T = n + m
    heads, d_spe = params.wq.shape[0], params.w_pe.shape[1]
    ws = [np.ascontiguousarray(w, np.float64) for w in (params.w_pe, params.wq, params.wk, params.wv, params.wo)]
    out = np.zeros((T, d_spe), np.float32)
    lam = np.zeros(T) if want_eigen else None
    U = np.zeros((T, T)) if want_eigen else None
    t64 = np.zeros((T, d_spe)) if want_eigen else None
    ptr = lambda a: a.ctypes.data if a is not None else None  # noqa: E731
    _check(load().aecct_spe_table(H.ctypes.data, n, n - m, d_spe, heads, *[w.ctypes.data for w in ws], out.ctypes.data,
                                  ptr(lam), ptr(U), ptr(t64)), "aecct_spe_table")
    return (out, t64, lam, U) if want_eigen else out
