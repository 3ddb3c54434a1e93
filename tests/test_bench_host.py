"""Host-side arithmetic of bench.py's roofline (no GPU).

The algorithmic fp32 operation count that the ALU roofline divides by is checked against its
closed form (66 d + 26 per block and token for AAP linears with ReLU, and the HPSA term over the
key counts), with the key counts taken by brute force from the oracle's HPSA masks (Sec. 4.2)
rather than from the degree sums bench.py uses.  The DRAM record is only used while the kernel
sources hash to the ones it was measured on.
"""
import numpy as np
import pytest

import bench
from oracle import oracle as O
from paper_2410_05911_gb300 import inputs as I


@pytest.mark.parametrize("key,mask_mode", [("polar64_32", 0), ("bch31_16", 0), ("bch63_36", 0), ("polar64_32", 1)])
def test_alu_ops_closed_form_with_mask_key_counts(key, mask_mode):
    w = I.workload(key)
    model = I.workload_model(key)
    model.mask_mode = mask_mode
    H = w.code.H
    m, n = H.shape
    T, d, N = n + m, model.d, model.n_layers
    dh = d // model.heads
    M1, M2 = O.masks(H)
    k1, k2 = int(M1.sum()), int(M2.sum())
    if mask_mode == 1:
        keys = model.heads * int((M1 | M2).sum())
    else:
        keys = model.h_first * k1 + (model.heads - model.h_first) * k2
    per_layer = T * (66 * d + 26) + keys * (2 * dh + 16) + T * model.heads * (dh + 1)
    head = T * (d - model.d_spe) + T * (2 * d + 1) + n * (T + 1) + n
    assert bench.alu_ops_per_word(w.code, model) == N * per_layer + head


def test_polar_alu_ops_figure():
    # the per-word figure the ALU roofline of the headline workload is quoted with
    w = I.workload("polar64_32")
    ops = bench.alu_ops_per_word(w.code, I.workload_model("polar64_32"))
    assert abs(ops / 1e6 - 7.33) < 0.005


def test_traffic_record_gated_on_kernel_sources_and_batch(monkeypatch, tmp_path):
    import json
    os_ = __import__("os")
    os_.makedirs(tmp_path / "profiles")
    rec = dict(workload="bch63_36", batch=262144, dram_bytes_read=9.0e6, dram_bytes_write=1.0e6, sources_sha256="a" * 64)
    with open(tmp_path / "profiles" / "aecct_decoder_kernel128_bch63_36_dram.json", "w") as f:
        json.dump(rec, f)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    monkeypatch.setattr(bench, "kernel_sources_digest", lambda: "a" * 64)
    assert bench.measured_traffic("bch63_36", 262144) == 10.0e6
    assert bench.measured_traffic("bch63_36", 4096) is None      # another batch: not scaled
    assert bench.measured_traffic("polar64_32", 65536) is None   # no record for this workload
    monkeypatch.setattr(bench, "kernel_sources_digest", lambda: "0" * 64)
    assert bench.measured_traffic("bch63_36", 262144) is None    # the kernel changed since
