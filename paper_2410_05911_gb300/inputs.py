"""Seeded synthetic inputs for the AECCT decoder: codes, channel outputs, model tensors.

This module is shared by the CUDA path's tests and benchmark and by the CPU
oracle's tests.  It holds none of the decoder's arithmetic: no syndrome, no
quantizer, no mask, no attention.  It only builds the problem instance the paper
sets up in Sec. 3 ("Problem Settings"):

* a binary linear code given by its parity-check matrix H ((n-k) x n over GF(2))
  and a generator G with G H^T = 0;
* messages, codewords, BPSK symbols x_s = 1 - 2x and AWGN channel outputs
  y = x_s + eps at a normalised SNR Eb/N0;
* a set of model tensors shaped like a trained AECCT (ternary in-block weights with
  a per-tensor scale, embeddings, LayerNorm parameters, output head).

The paper's parity-check matrices (taken from a public code database) and its
trained weights are not available, so codes are constructed from their textbook
definitions (BCH from the generator polynomial, Polar from the Arikan kernel with a
Bhattacharyya-ordered frozen set, regular LDPC from a seeded socket permutation) and
the weights are drawn at random with the zero fraction and scale that the paper's
ternary quantizer (Sec. 4.1, eq. Ternary) yields on Gaussian weights.

All randomness comes from numpy's PCG64 generator seeded explicitly.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Dict, List, Optional

import numpy as np

# ----------------------------------------------------------------------------
# GF(2) helpers (plain linear algebra over the two-element field)
# ----------------------------------------------------------------------------


def gf2_rank(A: np.ndarray) -> int:
    """Rank of a 0/1 matrix over GF(2) by Gaussian elimination."""
    M = (np.array(A, dtype=np.uint8) & 1).copy()
    rows, cols = M.shape
    r = 0
    for c in range(cols):
        piv = None
        for i in range(r, rows):
            if M[i, c]:
                piv = i
                break
        if piv is None:
            continue
        if piv != r:
            M[[r, piv]] = M[[piv, r]]
        for i in range(rows):
            if i != r and M[i, c]:
                M[i] ^= M[r]
        r += 1
        if r == rows:
            break
    return r


def gf2_nullspace(H: np.ndarray) -> np.ndarray:
    """Basis (rows) of {c : H c = 0 mod 2}."""
    M = (np.array(H, dtype=np.uint8) & 1).copy()
    rows, cols = M.shape
    pivots: List[int] = []
    r = 0
    for c in range(cols):
        piv = None
        for i in range(r, rows):
            if M[i, c]:
                piv = i
                break
        if piv is None:
            continue
        if piv != r:
            M[[r, piv]] = M[[piv, r]]
        for i in range(rows):
            if i != r and M[i, c]:
                M[i] ^= M[r]
        pivots.append(c)
        r += 1
        if r == rows:
            break
    free = [c for c in range(cols) if c not in set(pivots)]
    basis = np.zeros((len(free), cols), dtype=np.uint8)
    for bi, f in enumerate(free):
        basis[bi, f] = 1
        for ri, pc in enumerate(pivots):
            if M[ri, f]:
                basis[bi, pc] = 1
    return basis


def _poly_mul_gf2(a: List[int], b: List[int]) -> List[int]:
    out = [0] * (len(a) + len(b) - 1)
    for i, ai in enumerate(a):
        if ai:
            for j, bj in enumerate(b):
                if bj:
                    out[i + j] ^= 1
    return out


def _poly_divmod_gf2(num: List[int], den: List[int]):
    num = list(num)
    dd = len(den) - 1
    while dd > 0 and den[dd] == 0:
        dd -= 1
    q = [0] * max(1, len(num) - dd)
    for i in range(len(num) - 1, dd - 1, -1):
        if num[i]:
            q[i - dd] = 1
            for j in range(dd + 1):
                num[i - dd + j] ^= den[j]
    return q, num[:dd]


# ----------------------------------------------------------------------------
# Code constructions
# ----------------------------------------------------------------------------


@dataclasses.dataclass
class LinearCode:
    """A binary linear code: H is (n-k) x n, G is k' x n with G H^T = 0 (mod 2)."""

    name: str
    n: int
    k: int
    H: np.ndarray  # uint8 [(n-k), n]
    G: np.ndarray  # uint8 [k', n]; k' = n - rank(H) >= k

    @property
    def m(self) -> int:
        return self.n - self.k

    @property
    def T(self) -> int:
        """Number of decoder tokens, 2n - k (Sec. 3)."""
        return 2 * self.n - self.k


def _gf2m_tables(m: int, prim: int):
    """exp/log tables of GF(2^m) built from a primitive polynomial (bitmask)."""
    q = 1 << m
    exp = [0] * (2 * q)
    log = [0] * q
    v = 1
    for i in range(q - 1):
        exp[i] = v
        log[v] = i
        v <<= 1
        if v & q:
            v ^= prim
    for i in range(q - 1, 2 * q):
        exp[i] = exp[i - (q - 1)]
    return exp, log


def _minimal_poly(m: int, prim: int, i: int) -> List[int]:
    """Minimal polynomial over GF(2) of alpha^i in GF(2^m) (coefficients low->high)."""
    exp, log = _gf2m_tables(m, prim)
    n = (1 << m) - 1
    coset = []
    j = i % n
    while j not in coset:
        coset.append(j)
        j = (2 * j) % n
    # product of (x - alpha^c) with coefficients in GF(2^m)
    poly = [1]  # field elements, low->high
    for c in coset:
        root = exp[c]
        new = [0] * (len(poly) + 1)
        for d, a in enumerate(poly):
            new[d + 1] ^= a  # a * x
            if a:
                new[d] ^= exp[(log[a] + log[root]) % n]  # a * root (char 2: minus == plus)
        poly = new
    assert all(a in (0, 1) for a in poly), "minimal polynomial must have binary coefficients"
    return poly


def bch_code(n: int, t_design: int, m: int, prim: int, name: Optional[str] = None) -> LinearCode:
    """Narrow-sense primitive BCH code of length n = 2^m - 1 and designed distance 2t+1.

    g(x) = lcm of the minimal polynomials of alpha^1 .. alpha^(2t); H is built from the
    parity polynomial h(x) = (x^n + 1) / g(x): row i holds x^i * h*(x), where h* is the
    reciprocal of h.  G holds the shifts x^i g(x).
    """
    assert n == (1 << m) - 1
    g = [1]
    seen = set()
    for i in range(1, 2 * t_design + 1):
        mp = tuple(_minimal_poly(m, prim, i))
        if mp in seen:
            continue
        seen.add(mp)
        g = _poly_mul_gf2(g, list(mp))
    deg_g = len(g) - 1
    k = n - deg_g
    xn1 = [1] + [0] * (n - 1) + [1]
    h, rem = _poly_divmod_gf2(xn1, g)
    assert not any(rem), "g(x) must divide x^n + 1"
    h = h[: k + 1]
    G = np.zeros((k, n), dtype=np.uint8)
    for i in range(k):
        G[i, i : i + deg_g + 1] = g
    hrec = h[::-1]
    H = np.zeros((n - k, n), dtype=np.uint8)
    for i in range(n - k):
        H[i, i : i + k + 1] = hrec
    return LinearCode(name or f"BCH({n},{k})", n, k, H, G)


def polar_code(n: int, k: int, design_ebn0_db: float = 0.0, name: Optional[str] = None) -> LinearCode:
    """Polar code from the Arikan kernel F = [[1,0],[1,1]], G_N = F^{(x)m} (no bit reversal).

    The frozen set holds the n-k bit-channels with the largest Bhattacharyya parameter,
    computed by the recursion Z_2M[j] = 2z - z^2, Z_2M[j+M] = z^2 (z = Z_M[j]) from
    z0 = exp(-R * 10^(EbN0/10)), ties broken toward the lower index.  H = G_N[:, frozen]^T.
    """
    m = int(round(math.log2(n)))
    assert 1 << m == n
    F = np.array([[1, 0], [1, 1]], dtype=np.uint8)
    GN = np.array([[1]], dtype=np.uint8)
    for _ in range(m):
        GN = np.kron(F, GN) % 2
    rate = k / n
    Z = [math.exp(-rate * 10 ** (design_ebn0_db / 10))]
    while len(Z) < n:
        M = len(Z)
        nz = [0.0] * (2 * M)
        for j, z in enumerate(Z):
            nz[j] = 2 * z - z * z
            nz[j + M] = z * z
        Z = nz
    order = sorted(range(n), key=lambda j: (-Z[j], j))
    frozen = sorted(order[: n - k])
    info = sorted(order[n - k :])
    H = GN[:, frozen].T.copy().astype(np.uint8)
    G = GN[info, :].copy().astype(np.uint8)
    code = LinearCode(name or f"Polar({n},{k})", n, k, H, G)
    code.frozen = frozen  # type: ignore[attr-defined]
    code.GN = GN  # type: ignore[attr-defined]
    return code


def ldpc_regular_code(n: int, k: int, dv: int, dc: int, seed: int, name: Optional[str] = None) -> LinearCode:
    """Random (dv, dc)-regular LDPC parity-check matrix from a seeded socket permutation.

    Each variable node gets dv sockets and each check node dc sockets; a uniformly random
    permutation matches them.  A draw with a repeated (check, variable) edge is redrawn.
    G is a basis of the GF(2) null space of H (H may be rank deficient).
    """
    m = n - k
    assert n * dv == m * dc, "regularity requires n*dv == (n-k)*dc"
    rng = np.random.Generator(np.random.PCG64(seed))
    var_sockets = np.repeat(np.arange(n), dv)
    chk_sockets = np.repeat(np.arange(m), dc)
    for _attempt in range(10000):
        perm = rng.permutation(len(var_sockets))
        chk = chk_sockets[perm]
        pairs = chk.astype(np.int64) * n + var_sockets
        if len(np.unique(pairs)) == len(pairs):
            H = np.zeros((m, n), dtype=np.uint8)
            H[chk, var_sockets] = 1
            G = gf2_nullspace(H)
            return LinearCode(name or f"LDPC({n},{k})", n, k, H, G)
    raise RuntimeError("could not draw a simple regular bipartite graph")


# ----------------------------------------------------------------------------
# Channel
# ----------------------------------------------------------------------------


def awgn_sigma(ebn0_db: float, rate: float) -> float:
    """Noise std for unit-energy BPSK at normalised SNR Eb/N0: (2 R 10^(EbN0/10))^(-1/2)."""
    return 1.0 / math.sqrt(2.0 * rate * 10 ** (ebn0_db / 10.0))


@dataclasses.dataclass
class ChannelBatch:
    codewords: np.ndarray  # uint8 [B, n]
    y: np.ndarray  # float32 [B, n]
    ebn0_db: float
    sigma: float


def channel_batch(code: LinearCode, B: int, ebn0_db: float, seed: int) -> ChannelBatch:
    """Uniform random messages -> codewords x (via G) -> BPSK x_s = 1 - 2x -> y = x_s + eps."""
    rng = np.random.Generator(np.random.PCG64(seed))
    kk = code.G.shape[0]
    msgs = rng.integers(0, 2, size=(B, kk), dtype=np.uint8)
    # GF(2) product in chunks (int32 accumulate, then parity)
    cw = np.empty((B, code.n), dtype=np.uint8)
    Gi = code.G.astype(np.int32)
    step = 8192
    for s in range(0, B, step):
        cw[s : s + step] = ((msgs[s : s + step].astype(np.int32) @ Gi) & 1).astype(np.uint8)
    sigma = awgn_sigma(ebn0_db, code.k / code.n)
    xs = 1.0 - 2.0 * cw.astype(np.float32)
    noise = rng.standard_normal(size=(B, code.n), dtype=np.float32) * np.float32(sigma)
    y = (xs + noise).astype(np.float32)
    return ChannelBatch(cw, y, ebn0_db, sigma)


# ----------------------------------------------------------------------------
# Synthetic model tensors
# ----------------------------------------------------------------------------

GEMM_NAMES = ("q", "k", "v", "o", "ffn1", "ffn2")


@dataclasses.dataclass
class ModelTensors:
    """Parameters of an AECCT decoder (inference form).

    w_tern[l][g] is int8 in {-1,0,1} with shape [d_out, d_in] (row = output unit) for
    g in (q, k, v, o, ffn1, ffn2); w_scale[l][g] is the per-tensor fp32 scale.
    """

    n: int
    k: int
    d: int
    n_layers: int
    heads: int
    h_first: int
    d_spe: int
    ffn_mult: int
    activation: int  # 0 = ReLU, 1 = GELU (erf)
    H: np.ndarray
    emb: np.ndarray  # [T, d - d_spe]
    spe: np.ndarray  # [T, d_spe]
    w_tern: List[List[np.ndarray]]
    w_scale: np.ndarray  # [n_layers, 6]
    bias: List[List[np.ndarray]]
    ln_gamma: np.ndarray  # [n_layers, 2, d]
    ln_beta: np.ndarray  # [n_layers, 2, d]
    w_d1: np.ndarray  # [d]
    b_d1: float
    w_out: np.ndarray  # [T, n]
    b_out: np.ndarray  # [n]
    ln_eps: float = 1e-5
    alpha_floor: float = 1e-5
    mask_mode: int = 0  # 0 = HPSA rings (Sec. 4.2); 1 = ECCT code-aware mask for all heads (Sec. 3)
    alpha_mode: int = 0  # 0 = one absmax alpha per token (C-1); 1 = one per quantised matrix of a word
    linear_mode: int = 0  # 0 = AAP ternary linears (Sec. 4.1); 1 = full-precision linears (ECCT, Sec. 3)
    w_full: Optional[List[List[np.ndarray]]] = None  # linear_mode 1: fp32 weights, same order as w_tern

    @property
    def T(self) -> int:
        return 2 * self.n - self.k

    def gemm_shape(self, g: int):
        d, F = self.d, self.ffn_mult * self.d
        return {0: (d, d), 1: (d, d), 2: (d, d), 3: (d, d), 4: (F, d), 5: (d, F)}[g]


def _inv_norm_cdf(p: float) -> float:
    # bisection on erf; only used to pick a scale constant
    lo, hi = -10.0, 10.0
    for _ in range(200):
        mid = 0.5 * (lo + hi)
        if 0.5 * (1 + math.erf(mid / math.sqrt(2))) < p:
            lo = mid
        else:
            hi = mid
    return 0.5 * (lo + hi)


def ternary_scale_for_zero_fraction(zero_frac: float, d_in: int) -> float:
    """Scale gamma*delta that a ternary quantizer with threshold at half the scale gives on
    N(0, 1/d_in) weights when a fraction `zero_frac` of them rounds to zero: a weight is
    zero iff |W| < scale/2, so scale = 2 * sigma * Phi^-1((1 + zero_frac)/2)."""
    sigma = 1.0 / math.sqrt(d_in)
    return 2.0 * sigma * _inv_norm_cdf(0.5 * (1.0 + zero_frac))


@dataclasses.dataclass
class SpeParams:
    """Parameters of the spectral positional encoding (Sec. 4.3): W_{2->d_SPE} and the SPE's
    multi-head self-attention projections (standard form, no biases)."""
    w_pe: np.ndarray   # [2, d_spe]
    wq: np.ndarray     # [heads, d_spe, d_e]
    wk: np.ndarray     # [heads, d_spe, d_e]
    wv: np.ndarray     # [heads, d_spe, d_e]
    wo: np.ndarray     # [d_spe, d_spe]


def spe_params(H: np.ndarray, d_spe: int, seed: int, heads: int = 4) -> SpeParams:
    """Seeded SPE parameters standing in for learned ones (float64).  The eigenvalue row of
    W_{2->d_SPE} is scaled by 1 / (2 max degree), a bound on the Laplacian's largest eigenvalue,
    and the eigenvector row by sqrt(T) (eigenvector entries are about 1/sqrt(T)), so that both
    columns of Phi contribute O(1) values; the projections are N(0, 1/d_SPE)."""
    if d_spe % heads:
        raise ValueError("d_spe must be a multiple of the SPE heads")
    m, n = H.shape
    T = n + m
    deg = max(int((H != 0).sum(0).max()), int((H != 0).sum(1).max()))
    rng = np.random.Generator(np.random.PCG64(seed))
    d_e = d_spe // heads
    w_pe = rng.standard_normal((2, d_spe))
    w_pe[0] /= 2.0 * deg
    w_pe[1] *= math.sqrt(T)
    s = 1.0 / math.sqrt(d_spe)
    wq = rng.standard_normal((heads, d_spe, d_e)) * s
    wk = rng.standard_normal((heads, d_spe, d_e)) * s
    wv = rng.standard_normal((heads, d_spe, d_e)) * s
    wo = rng.standard_normal((d_spe, d_spe)) * s
    return SpeParams(w_pe, wq, wk, wv, wo)


_SPE_CACHE: Dict[tuple, np.ndarray] = {}


def spe_for_code(H: np.ndarray, d_spe: int, seed: int) -> np.ndarray:
    """The model's SPE table: the host precompute of Sec. 4.3 (paper_2410_05911_gb300.spe) on
    seeded SPE parameters, cached per (H, d_spe, seed) within the process."""
    if d_spe == 0:
        return np.zeros((H.shape[0] + H.shape[1], 0), np.float32)
    key = (H.shape, H.tobytes(), d_spe, seed)
    if key not in _SPE_CACHE:
        from . import spe

        _SPE_CACHE[key] = spe.spe_table(H, spe_params(H, d_spe, seed))
    return _SPE_CACHE[key].copy()


def random_model(
    code: LinearCode,
    d: int,
    n_layers: int,
    seed: int,
    heads: int = 8,
    h_first: Optional[int] = None,
    d_spe: Optional[int] = None,
    zero_frac: float = 0.5,
    activation: int = 0,
    ffn_mult: int = 4,
    zero_weights: bool = False,
    binary: bool = False,
    full_precision: bool = False,
    spe_noise: bool = False,
) -> ModelTensors:
    """Seeded synthetic AECCT parameters shaped like a trained model.

    Ternary weights: exactly round(zero_frac * size) zeros per tensor at random positions,
    the rest +1/-1 with equal probability; the scale is the one the paper's quantizer
    would produce on N(0, 1/d_in) weights at that zero fraction, times a per-tensor jitter
    in [0.9, 1.1].  Biases and LayerNorm parameters are small random values so that an
    indexing mistake changes the output.  The SPE table is the Tanner-graph spectral encoding
    of Sec. 4.3 computed on the host from H with seeded SPE parameters (spe_for_code); at
    inference it is a fixed table.

    binary=True draws the binary-weight variant (App. D): every weight is +1 or -1 and the
    per-tensor scale is the mean |W| of N(0, 1/d_in) weights, sqrt(2 / (pi d_in)), times the
    same jitter.

    full_precision=True also draws fp32 weights W ~ N(0, 1/d_in) per tensor (the full-precision
    linear layers of the ECCT baseline, Sec. 3) and selects them (linear_mode = 1).

    spe_noise=True draws the SPE table as seeded N(0, 1) values instead (for shape tests of the
    decoder at its largest token counts, where the O(T^3) precompute would dominate and the
    table's content plays no role).
    """
    rng = np.random.Generator(np.random.PCG64(seed))
    T = code.T
    if h_first is None:
        h_first = heads // 2
    if d_spe is None:
        d_spe = d // 4
    F = ffn_mult * d
    shapes = [(d, d), (d, d), (d, d), (d, d), (F, d), (d, F)]
    w_tern: List[List[np.ndarray]] = []
    bias: List[List[np.ndarray]] = []
    w_scale = np.zeros((n_layers, 6), dtype=np.float32)
    w_full: Optional[List[List[np.ndarray]]] = [] if full_precision else None
    for l in range(n_layers):
        wl, bl, fl = [], [], []
        for g, (dout, din) in enumerate(shapes):
            size = dout * din
            if zero_weights:
                t = np.zeros(size, dtype=np.int8)
            elif binary:
                t = rng.choice(np.array([-1, 1], dtype=np.int8), size=size)
            else:
                nz = int(round(zero_frac * size))
                t = rng.choice(np.array([-1, 1], dtype=np.int8), size=size)
                zpos = rng.permutation(size)[:nz]
                t[zpos] = 0
            wl.append(t.reshape(dout, din))
            base = math.sqrt(2.0 / (math.pi * din)) if binary else ternary_scale_for_zero_fraction(zero_frac, din)
            w_scale[l, g] = base * rng.uniform(0.9, 1.1)
            bl.append((0.1 * rng.standard_normal(dout)).astype(np.float32))
            if full_precision:
                fl.append((rng.standard_normal((dout, din)) / math.sqrt(din)).astype(np.float32))
        w_tern.append(wl)
        bias.append(bl)
        if full_precision:
            w_full.append(fl)
    ln_gamma = (1.0 + 0.1 * rng.standard_normal((n_layers, 2, d))).astype(np.float32)
    ln_beta = (0.1 * rng.standard_normal((n_layers, 2, d))).astype(np.float32)
    emb = rng.standard_normal((T, d - d_spe)).astype(np.float32)
    spe = (rng.standard_normal((T, d_spe)).astype(np.float32) if spe_noise
           else spe_for_code(code.H, d_spe, seed + 7919))
    w_d1 = (rng.standard_normal(d) / math.sqrt(d)).astype(np.float32)
    b_d1 = float(np.float32(0.1 * rng.standard_normal()))
    w_out = (2.0 * rng.standard_normal((T, code.n)) / math.sqrt(T)).astype(np.float32)
    b_out = (0.1 * rng.standard_normal(code.n)).astype(np.float32)
    return ModelTensors(
        n=code.n, k=code.k, d=d, n_layers=n_layers, heads=heads, h_first=h_first, d_spe=d_spe,
        ffn_mult=ffn_mult, activation=activation, H=code.H.copy(), emb=emb, spe=spe,
        w_tern=w_tern, w_scale=w_scale, bias=bias, ln_gamma=ln_gamma, ln_beta=ln_beta,
        w_d1=w_d1, b_d1=b_d1, w_out=w_out, b_out=b_out,
        linear_mode=1 if full_precision else 0, w_full=w_full,
    )


# ----------------------------------------------------------------------------
# The five workloads (code, model shape, batch, Eb/N0 points)
# ----------------------------------------------------------------------------


@dataclasses.dataclass
class Workload:
    key: str
    code: LinearCode
    d: int
    n_layers: int
    batch: int
    ebn0_db: tuple
    zero_frac: float
    seed: int


_CODE_CACHE: Dict[str, LinearCode] = {}


def make_code(key: str) -> LinearCode:
    if key in _CODE_CACHE:
        return _CODE_CACHE[key]
    if key == "bch31_16":
        c = bch_code(31, 3, 5, 0b100101)  # x^5 + x^2 + 1
    elif key == "polar64_32":
        c = polar_code(64, 32, 0.0)
    elif key == "ldpc128_64":
        c = ldpc_regular_code(128, 64, 3, 6, seed=12864)
    elif key == "bch63_36":
        c = bch_code(63, 5, 6, 0b1000011)  # x^6 + x + 1
    elif key == "ldpc384_192":
        c = ldpc_regular_code(384, 192, 3, 6, seed=384192)
    elif key == "hamming7_4":
        H = np.array([[1, 0, 1, 0, 1, 0, 1], [0, 1, 1, 0, 0, 1, 1], [0, 0, 0, 1, 1, 1, 1]], dtype=np.uint8)
        c = LinearCode("Hamming(7,4)", 7, 4, H, gf2_nullspace(H))
    else:
        raise KeyError(key)
    _CODE_CACHE[key] = c
    return c


WORKLOADS = {
    "bch31_16": dict(code="bch31_16", d=32, n_layers=2, batch=1024, ebn0_db=(4.0,), zero_frac=0.5, seed=1),
    "polar64_32": dict(code="polar64_32", d=64, n_layers=6, batch=65536, ebn0_db=(4.0, 5.0, 6.0), zero_frac=0.4, seed=2),
    "ldpc128_64": dict(code="ldpc128_64", d=128, n_layers=6, batch=131072, ebn0_db=(3.0,), zero_frac=0.5, seed=3),
    "bch63_36": dict(code="bch63_36", d=128, n_layers=10, batch=262144, ebn0_db=(4.0, 5.0, 6.0, 7.0), zero_frac=0.5, seed=4),
    "ldpc384_192": dict(code="ldpc384_192", d=128, n_layers=6, batch=16384, ebn0_db=(2.5,), zero_frac=0.5, seed=5),
}


def workload(key: str) -> Workload:
    w = WORKLOADS[key]
    return Workload(key, make_code(w["code"]), w["d"], w["n_layers"], w["batch"], tuple(w["ebn0_db"]), w["zero_frac"], w["seed"])


def workload_model(key: str, **overrides) -> ModelTensors:
    w = workload(key)
    kw = dict(zero_frac=w.zero_frac)
    kw.update(overrides)
    return random_model(w.code, w.d, w.n_layers, seed=1000 + w.seed, **kw)
