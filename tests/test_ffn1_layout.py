"""The d = 128 layout of FFN1's accumulators and FFN2's operand in tensor memory.

FFN1's output column c holds hidden unit ffn1_unit_of_column(D, c) (aecct_internal.h): the weight
stream puts that unit's weight row at column c.  Each thread of a row owns one column slice s of
the hidden units, [128 s, 128 s + 128), handled in four chunks of 32 units in order; after the row
maximum it writes the codes of unit h, two to a 32-bit column, to column h / 2, which is the
K order FFN2's MMA reads its A operand in.  Nothing orders the threads of one row between those
reads and writes, so a code column must be one that the same thread has already read.  These
tests check the map from the header itself (compiled by g++) against those requirements; no GPU.
"""
import os
import subprocess

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2410_05911_gb300", "csrc")
CUDA_INC = os.path.join(os.environ.get("CUDA_HOME", "/usr/local/cuda"), "include")

HARNESS = r"""
#include "aecct_internal.h"
#include <cstdio>
int main() {
  for (int D : {32, 64, 128})
    for (int c = 0; c < 4 * D; ++c) std::printf("%d %d %d\n", D, c, aecct::ffn1_unit_of_column(D, c));
  return 0;
}
"""


@pytest.fixture(scope="module")
def unit_of_column(tmp_path_factory):
    if not os.path.isdir(CUDA_INC):
        pytest.skip("CUDA headers not found")
    d = tmp_path_factory.mktemp("ffn1_layout")
    src, exe = d / "harness.cpp", d / "harness"
    src.write_text(HARNESS)
    subprocess.run(["g++", "-std=c++17", "-O1", f"-I{CUDA_INC}", f"-I{CSRC}", str(src), "-o", str(exe)], check=True)
    out = subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout
    table = {}
    for line in out.split("\n"):
        if line.strip():
            D, c, u = map(int, line.split())
            table.setdefault(D, []).append(u)
    return {D: np.array(v) for D, v in table.items()}


def test_identity_below_128(unit_of_column):
    for D in (32, 64):
        assert (unit_of_column[D] == np.arange(4 * D)).all()


def test_d128_is_a_permutation(unit_of_column):
    u = unit_of_column[128]
    assert u.shape == (512,)
    assert (np.sort(u) == np.arange(512)).all()


def test_d128_slice_ownership_and_first_tile_pair(unit_of_column):
    u = unit_of_column[128]
    col_of = np.empty(512, dtype=int)
    col_of[u] = np.arange(512)
    for s in range(4):
        units = np.arange(128 * s, 128 * s + 128)
        # the first 64 units in [64 s, 64 s + 64), the other 64 in [256 + 64 s, 256 + 64 s + 64), in order
        assert (col_of[units[:64]] == 64 * s + np.arange(64)).all()
        assert (col_of[units[64:]] == 256 + 64 * s + np.arange(64)).all()
    # FFN1's first N-tile pair (columns [0, 256)) holds the first half of every slice's units
    first = set(u[:256].tolist())
    assert first == {128 * s + j for s in range(4) for j in range(64)}


def test_d128_codes_compact_in_place_within_each_thread(unit_of_column):
    u = unit_of_column[128]
    col_of = np.empty(512, dtype=int)
    col_of[u] = np.arange(512)
    for s in range(4):
        read = set()
        for ch in range(4):
            chunk = np.arange(128 * s + 32 * ch, 128 * s + 32 * ch + 32)
            read |= set(col_of[chunk].tolist())  # the chunk's values are read first
            code_cols = set((chunk // 2).tolist())
            # codes go only to columns this thread has already read, inside its own first range
            assert code_cols <= read, (s, ch)
            assert all(64 * s <= c < 64 * s + 64 for c in code_cols)
    # every unit's code in column h / 2: FFN2's operand is [0, 256) in natural K order, clear of its
    # accumulators [256, 384)
    codes = np.arange(512) // 2
    assert codes.min() == 0 and codes.max() == 255
