"""CPU-side checks of the C ABI: the library builds and loads, exports every function that
include/aecct.h declares, packs weights in the documented 2-bit format, and rejects invalid
model descriptions before touching a GPU."""
import copy
import os
import re

import numpy as np
import pytest

from paper_2410_05911_gb300 import aecct as A
from paper_2410_05911_gb300 import inputs as I

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def header_functions():
    text = open(os.path.join(ROOT, "include", "aecct.h")).read()
    return sorted(set(re.findall(r"^\s*(?:int|const char \*)\s*(aecct_\w+)\s*\(", text, re.M)))


def test_library_exports_every_declared_function():
    L = A.load()
    names = header_functions()
    assert len(names) >= 11
    for name in names:
        assert hasattr(L, name), name
    assert set(names) == set(A.EXPORTED_SYMBOLS)


def test_status_strings():
    assert A.status_string(0) == "ok"
    assert "timed out" in A.status_string(A.AECCT_ERR_TIMEOUT)
    assert A.status_string(-99) == "unknown status"


def test_pack_ternary_layout():
    t = np.array([[1, 0, -1, 1, 0, 0, 0, -1]], np.int8)
    p = A.pack_ternary(t)
    assert p.tolist() == [[0b01110001, 0b11000000]]
    rng = np.random.default_rng(0)
    t = rng.integers(-1, 2, (16, 64)).astype(np.int8)
    p = A.pack_ternary(t)
    codes = np.stack([(p >> (2 * s)) & 3 for s in range(4)], -1).reshape(16, 64)
    back = np.where(codes == 1, 1, np.where(codes == 3, -1, 0))
    assert (back == t).all() and not (codes == 2).any()
    with pytest.raises(ValueError):
        A.pack_ternary(np.array([[2, 0, 0, 0]], np.int8))


def _status(model, **kw):
    st, h = A.create_handle(model, **kw)
    assert h is None or st == 0
    return st


@pytest.mark.parametrize("mutate,expected", [
    (lambda m: setattr(m, "h_first", 9), A.AECCT_ERR_INVALID_ARG),
    (lambda m: setattr(m, "h_first", -1), A.AECCT_ERR_INVALID_ARG),
    (lambda m: setattr(m, "d_spe", 32), A.AECCT_ERR_INVALID_ARG),
    (lambda m: setattr(m, "n_layers", 0), A.AECCT_ERR_INVALID_ARG),
    (lambda m: setattr(m, "ln_eps", float("nan")), A.AECCT_ERR_INVALID_ARG),
    (lambda m: setattr(m, "alpha_floor", 0.0), A.AECCT_ERR_INVALID_ARG),
    (lambda m: m.H.__setitem__((0, 0), 2), A.AECCT_ERR_INVALID_ARG),
    (lambda m: m.H.__setitem__((0, slice(None)), 0), A.AECCT_ERR_INVALID_ARG),
    (lambda m: m.H.__setitem__((slice(None), 3), 0), A.AECCT_ERR_INVALID_ARG),
    (lambda m: setattr(m, "activation", 7), A.AECCT_ERR_INVALID_ARG),
    (lambda m: setattr(m, "mask_mode", 2), A.AECCT_ERR_INVALID_ARG),
    (lambda m: setattr(m, "mask_mode", -1), A.AECCT_ERR_INVALID_ARG),
    (lambda m: setattr(m, "alpha_mode", 2), A.AECCT_ERR_INVALID_ARG),
    (lambda m: setattr(m, "linear_mode", 2), A.AECCT_ERR_INVALID_ARG),
    (lambda m: setattr(m, "ffn_mult", 2), A.AECCT_ERR_UNSUPPORTED),
])
def test_create_rejects_invalid_descriptions(mutate, expected):
    m = copy.deepcopy(I.workload_model("bch31_16"))
    mutate(m)
    assert _status(m) == expected


def test_create_rejects_invalid_packed_code_and_shapes():
    m = I.workload_model("bch31_16")
    hm = A._HostModel(m)
    hm.w_packed[5] = 0b00100000  # code 10 in slot 2
    import ctypes
    h = ctypes.c_void_p()
    assert A.load().aecct_create(ctypes.byref(hm.desc), ctypes.byref(h)) == A.AECCT_ERR_INVALID_ARG
    # valid but outside this build: d = 48 with 8 heads
    code = I.make_code("bch31_16")
    m48 = I.random_model(code, 48, 1, seed=3, d_spe=8)
    assert _status(m48) == A.AECCT_ERR_UNSUPPORTED
    # a cluster size that cannot hold one codeword
    big = I.workload_model("ldpc384_192")
    assert _status(big, cluster_ctas=2) == A.AECCT_ERR_INVALID_ARG
    # attention modes: unknown value, and warp tasks where they do not apply (more than 128 token
    # rows once each node type starts on a 32-row boundary; d = 128 with one alpha per word)
    assert _status(I.workload_model("bch31_16"), attention_mode=4) == A.AECCT_ERR_INVALID_ARG
    # staged rows: d = 128 only, at most 640 token rows per group
    assert _status(I.workload_model("bch31_16"), attention_mode=3) == A.AECCT_ERR_UNSUPPORTED
    c680 = I.ldpc_regular_code(680, 340, 3, 6, seed=680340)
    assert _status(I.random_model(c680, 128, 1, seed=3, spe_noise=True), attention_mode=3) == A.AECCT_ERR_UNSUPPORTED
    assert _status(I.workload_model("ldpc128_64"), attention_mode=2) == A.AECCT_ERR_UNSUPPORTED
    m63 = copy.deepcopy(I.workload_model("bch63_36"))
    m63.alpha_mode = 1
    assert _status(m63, attention_mode=2) == A.AECCT_ERR_UNSUPPORTED
    # d = 128: T = 98 + 28 = 126 tokens, but the 98 variables take rows 0..97, so the checks would
    # start at row 128
    c98 = I.ldpc_regular_code(98, 70, 2, 7, seed=0)
    assert c98.n + c98.H.shape[0] <= 128
    assert _status(I.random_model(c98, 128, 1, seed=3), attention_mode=2) == A.AECCT_ERR_UNSUPPORTED
    # one alpha per word needs one CTA per word
    m2 = copy.deepcopy(I.workload_model("ldpc128_64"))
    m2.alpha_mode = 1
    assert _status(m2) == A.AECCT_ERR_UNSUPPORTED
    # NULL description / output pointer
    assert A.load().aecct_create(None, ctypes.byref(h)) == A.AECCT_ERR_INVALID_ARG
    assert A.load().aecct_create(ctypes.byref(hm.desc), None) == A.AECCT_ERR_INVALID_ARG


def test_full_precision_description_checks():
    import ctypes
    code = I.make_code("bch31_16")
    m = I.random_model(code, 32, 1, seed=4, full_precision=True)
    L = A.load()
    h = ctypes.c_void_p()
    # alpha belongs to the AAP quantiser: not with full-precision linears
    m1 = copy.deepcopy(m)
    m1.alpha_mode = 1
    assert _status(m1) == A.AECCT_ERR_INVALID_ARG
    # the fp32 weights are required, and must be finite
    hm = A._HostModel(m)
    hm.desc.w_full = None
    assert L.aecct_create(ctypes.byref(hm.desc), ctypes.byref(h)) == A.AECCT_ERR_INVALID_ARG
    hm = A._HostModel(m)
    hm.w_full[7] = np.float32(np.inf)
    assert L.aecct_create(ctypes.byref(hm.desc), ctypes.byref(h)) == A.AECCT_ERR_INVALID_ARG
    # the ternary arrays are not read: NULL is fine (create then goes on to the device checks)
    hm = A._HostModel(m)
    assert hm.desc.w_packed is None and hm.desc.w_scale is None


def test_calls_on_null_handle():
    L = A.load()
    assert L.aecct_decode(None, None, 1, None, None, None, None) == A.AECCT_ERR_INVALID_ARG
    assert L.aecct_synchronize(None) == A.AECCT_ERR_INVALID_ARG
    assert L.aecct_destroy(None) == A.AECCT_ERR_INVALID_ARG
    assert L.aecct_set_capture(None, 0, None, None, None, None) == A.AECCT_ERR_INVALID_ARG


def test_caller_outputs_are_checked_before_the_kernel_writes_them():
    torch = pytest.importorskip("torch")
    cpu = torch.device("cpu")
    B, n, m = 5, 31, 15
    ok = (torch.empty((B, n), dtype=torch.uint8), torch.empty((B, m), dtype=torch.uint8), None)
    assert A.check_outputs(ok, B, n, m, cpu)[0] is ok[0]
    assert A.check_outputs((ok[0], None, torch.empty((B, n))), B, n, m, cpu)[2].shape == (B, n)
    bad = [
        (None, None, None),                                                         # bits are required
        (torch.empty((B - 1, n), dtype=torch.uint8), None, None),                  # too few rows
        (torch.empty((B, n), dtype=torch.int32), None, None),                      # wrong type
        (ok[0], torch.empty((B, m + 1), dtype=torch.uint8), None),                 # syndrome too wide
        (ok[0], None, torch.empty((B, n), dtype=torch.float64)),                   # logits type
        (torch.empty((n, B), dtype=torch.uint8).t(), None, None),                  # not contiguous
        (ok[0].to("meta"), None, None),                                            # another device
    ]
    for out in bad:
        with pytest.raises(ValueError):
            A.check_outputs(out, B, n, m, cpu)


def test_aap_ternarize_rejects_bad_arguments_before_any_device_work():
    L = A.load()
    lens = np.array([8, 6], np.int64)  # 6 is not a multiple of 4
    deltas = np.ones(2, np.float32)
    P = 0x1000  # never dereferenced: the arguments are refused first
    assert L.aecct_aap_ternarize(P, 2, lens.ctypes.data, deltas.ctypes.data, 1e-8, P, P, None, None) == \
        A.AECCT_ERR_INVALID_ARG
    lens = np.array([8, 4], np.int64)
    assert L.aecct_aap_ternarize(P, 2, lens.ctypes.data, deltas.ctypes.data, 0.0, P, P, None, None) == \
        A.AECCT_ERR_INVALID_ARG  # eps must be > 0
    bad = np.array([1.0, -1.0], np.float32)
    assert L.aecct_aap_ternarize(P, 2, lens.ctypes.data, bad.ctypes.data, 1e-8, P, P, None, None) == \
        A.AECCT_ERR_INVALID_ARG  # delta must be > 0
    assert L.aecct_aap_ternarize(None, 2, lens.ctypes.data, deltas.ctypes.data, 1e-8, P, P, None, None) == \
        A.AECCT_ERR_INVALID_ARG
    assert L.aecct_aap_ternarize(None, 0, None, None, 1e-8, None, None, None, None) == A.AECCT_OK
