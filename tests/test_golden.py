"""The oracle against small examples worked by hand from the paper's definitions
(tests/golden/, each file names the passage it follows)."""
import os

import numpy as np

from oracle import oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _lines(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return [ln.split() for ln in f if ln.strip() and not ln.startswith("#")]


def test_hamming74_decisions_syndrome_and_masks():
    rows = _lines("hamming74_masks_syndrome.txt")
    H = np.array([[int(v) for v in r[1:]] for r in rows if r[0] == "H"], np.uint8)
    get = {r[0]: r[1:] for r in rows if r[0] in ("y", "bits", "syndrome", "tokens")}
    y = np.array(get["y"], np.float32)
    bits = O.hard_decision(y)
    assert bits.tolist() == [int(v) for v in get["bits"]]
    s = O.syndrome(H, bits)
    assert s.tolist() == [int(v) for v in get["syndrome"]]
    tokens = np.concatenate([np.abs(y), 1.0 - 2.0 * s.astype(np.float32)])
    assert np.allclose(tokens, np.array(get["tokens"], np.float32))
    M1, M2 = O.masks(H)
    for r in rows:
        if r[0] in ("M1", "M2"):
            t = int(r[1].rstrip(":"))
            M = M1 if r[0] == "M1" else M2
            assert np.flatnonzero(M[t]).tolist() == [int(v) for v in r[2:]], (r[0], t)


def test_quant_rows():
    rows = _lines("quant_rows.txt")
    for i in range(0, len(rows), 3):
        x = np.array(rows[i][1:], np.float32)
        q, alpha = O.quant_row(x)
        assert float(alpha) == float(rows[i + 1][1])
        assert q.tolist() == [int(v) for v in rows[i + 2][1:]]


def test_layernorm_row():
    rows = _lines("layernorm_row.txt")
    v = np.array(rows[0][1:], np.float32)
    for i in range(1, len(rows), 3):
        g = np.array(rows[i][1:], np.float32)
        b = np.array(rows[i + 1][1:], np.float32)
        want = np.array(rows[i + 2][1:], np.float64)
        got = O.layernorm_row(v, g, b, eps=0.0).astype(np.float64)
        assert np.allclose(got, want, rtol=1e-6, atol=1e-6)
