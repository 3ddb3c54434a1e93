"""Planted mistakes: the oracle's pins must catch each one.

Every entry below is a copy of oracle/aecct_oracle.c with one plausible mistake (a dropped term,
a wrong sign, index or constant, a transposed operand, a swapped mask), each against the passage
of the paper the mistake would break.  Mistakes that cannot change a result are not listed: the
clip of the codes at +-Q_b, for instance, never acts, since alpha is at least max |x|.

Each copy is compiled on its own and the pin suites (tests/test_oracle_pins.py,
tests/test_golden.py, tests/test_oracle_forward_f64.py) run against it in a subprocess.  The test
asserts that each copy fails a pin by an assertion, and that the unmodified source, compiled the
same way, passes them.  Nothing here touches a GPU.
"""
import os
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

from oracle import oracle as O

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "aecct_oracle.c")
PINS = ["tests/test_oracle_pins.py", "tests/test_golden.py", "tests/test_oracle_forward_f64.py"]

# (name, passage, original text, planted text); each original occurs once in the source
MUTANTS = [
    # Sec. 3: hard decisions, syndrome, tokens
    ("hard decision sign", "Sec. 3", "b[j] = (y[j] < 0.0f) ? 1 : 0;", "b[j] = (y[j] > 0.0f) ? 1 : 0;"),
    ("syndrome reads H transposed", "Sec. 3",
     "acc ^= (uint8_t)(H[(size_t)i * n + j] & b[j]);", "acc ^= (uint8_t)(H[(size_t)j * m + i] & b[j]);"),
    ("syndrome token s instead of 1 - 2s", "Sec. 3", "1.0f - 2.0f * (float)w->s[t - n]", "(float)w->s[t - n]"),
    ("magnitude token y instead of |y|", "Sec. 3", "fabsf(y[t])", "y[t]"),
    ("embedding row ignores the position", "Sec. 3 (ECCT)", "m->emb[(size_t)t * de + c]", "m->emb[c]"),
    ("SPE written over the embedding", "Sec. 4.3", "w->x[(size_t)t * d + de + c] = m->spe", "w->x[(size_t)t * d + c] = m->spe"),
    # Sec. 4.2: masks and HPSA
    ("first and second ring swapped", "Sec. 4.2", "(e < h_first ? M1 : M2)", "(e < h_first ? M2 : M1)"),
    ("first ring one-directional", "Sec. 4.2", "M1[(size_t)(n + i) * T + j] = 1;", ";"),
    ("second ring without the node itself", "Sec. 4.2",
     "M2[(size_t)a * T + b] = hit;", "M2[(size_t)a * T + b] = (uint8_t)(a != b && hit);"),
    ("check-check ring from the wrong H axis", "Sec. 4.2",
     "hit = H[(size_t)a * n + j] & H[(size_t)b * n + j];", "hit = H[(size_t)a * n + j] & H[(size_t)a * n + j];"),
    ("score scale 1/sqrt(d) instead of 1/sqrt(d_h)", "Sec. 4.2", "sqrt((double)dh)", "sqrt((double)d)"),
    ("score scale without log2(e)", "Sec. 4.2", "(float)(1.4426950408889634074 / sqrt", "(float)(1.0 / sqrt"),
    ("odd-feature chain dropped", "Sec. 4.2", "return de + dod;", "return de;"),
    ("softmax not normalised", "Sec. 4.2", "float inv = 1.0f / l;", "float inv = 1.0f;"),
    ("K used as V", "Sec. 4.2", "const float *vv = V + (size_t)u * d + e * dh;", "const float *vv = K + (size_t)u * d + e * dh;"),
    ("every head uses head 0's query", "Sec. 4.2", "const float *q = Q + (size_t)t * d + e * dh;", "const float *q = Q + (size_t)t * d;"),
    ("exp2 series drops a term", "Sec. 4.2", "for (int k = 6; k >= 0; --k)", "for (int k = 5; k >= 0; --k)"),
    ("exp2 coefficients off by one factorial", "Sec. 4.2", "term * ln2 / (double)(k + 1)", "term * ln2 / (double)(k + 2)"),
    # Sec. 4.1: Quant and AAPLinear
    ("Q_b = 128", "Sec. 4.1 eq. Quant", "float r = 127.0f / a;", "float r = 128.0f / a;"),
    ("truncation instead of rounding", "Sec. 4.1 eq. Quant", "float v = rintf(x[i] * r);", "float v = truncf(x[i] * r);"),
    ("absmax of signed values", "Sec. 4.1 eq. Quant", "float ax = fabsf(x[i]);", "float ax = x[i];"),
    ("alpha floor ignored", "Sec. 4.1 eq. Quant", "  if (!(a > alpha_floor)) a = alpha_floor;\n  quant_with_alpha",
     "  quant_with_alpha"),
    ("dequantisation without alpha", "Sec. 4.1 eq. AAPLinear", "float f = (s_w * alpha) / 127.0f;", "float f = s_w / 127.0f;"),
    ("dequantisation without the weight scale", "Sec. 4.1 eq. AAPLinear", "float f = (s_w * alpha) / 127.0f;",
     "float f = alpha / 127.0f;"),
    ("linear bias dropped", "Sec. 4.1 eq. AAPLinear", "out[o] = (float)acc * f + b[o];", "out[o] = (float)acc * f;"),
    ("weights transposed", "Sec. 4.1 eq. AAPLinear",
     "acc += (int32_t)q[i] * (int32_t)wr[i];", "acc += (int32_t)q[i] * (int32_t)W[(size_t)i * N + o];"),
    ("ternary percentile at the minimum", "Sec. 4.1 eq. Ternary", "double pos = 0.5 * (double)(len - 1);", "double pos = 0.0;"),
    ("ternary threshold without delta", "Sec. 4.1 eq. Ternary", "float sc = gamma * delta;", "float sc = gamma;"),
    # Sec. 5: Post-LN blocks, Sec. 4 item 4: FFN
    ("attention residual dropped", "Sec. 5",
     "w->v[c] = w->x[(size_t)t * d + c] + w->o[(size_t)t * d + c];", "w->v[c] = w->o[(size_t)t * d + c];"),
    ("FFN residual dropped", "Sec. 5", "w->v[c] = w->x[(size_t)t * d + c] + w->o[c];", "w->v[c] = w->o[c];"),
    ("LayerNorm variance over d - 1", "Sec. 5", "float var = oracle_psum(tmp, d) * inv_d;",
     "float var = oracle_psum(tmp, d) / (float)(d - 1);"),
    ("LayerNorm epsilon dropped", "Sec. 5", "sqrtf(var + eps)", "sqrtf(var)"),
    ("LayerNorm gamma and beta swapped", "Sec. 5", "* rstd) * g[i] + b[i];", "* rstd) * b[i] + g[i];"),
    ("pairwise sum drops the upper half", "Sec. 5", "  return a + b;\n}", "  return a + 0.0f * b;\n}"),
    ("ReLU dropped", "Sec. 4 item 4", "ur[c] = ur[c] > 0.0f ? ur[c] : 0.0f;", "ur[c] = ur[c];"),
    ("GELU coefficient sign", "Sec. 4 item 4 (GELU option)", "q = fmaf(q, t, -0.284496736f);", "q = fmaf(q, t, 0.284496736f);"),
    # Sec. 3: output head and decisions
    ("output-head bias b_d1 dropped", "Sec. 3 (ECCT)", "w->z[t] = oracle_psum(w->v, d) + m->b_d1;", "w->z[t] = oracle_psum(w->v, d);"),
    ("W_o read transposed", "Sec. 3 (ECCT)", "m->w_out[(size_t)t * n + j]", "m->w_out[(size_t)j * T + t]"),
    ("output bias b_o dropped", "Sec. 3 (ECCT)", "w->eps[j] = e + m->b_out[j];", "w->eps[j] = e;"),
    ("decision from eps alone", "Sec. 3", "(y[j] * w->eps[j] < 0.0f)", "(w->eps[j] < 0.0f)"),
    # Sec. 3: the ECCT baseline's mask and full-precision linears
    ("code-aware mask without the second ring", "Sec. 3 (ECCT)",
     "w->M1[i] = w->M2[i] = (uint8_t)(w->M1[i] | w->M2[i]);", "w->M2[i] = w->M1[i];"),
    ("bf16 rounding truncates", "Sec. 3 (ECCT, full precision)",
     "if (low > 0x8000u || (low == 0x8000u && (keep & 0x10000u))) keep += 0x10000u;", "(void)low;"),
    ("full-precision bias dropped", "Sec. 3 (ECCT, full precision)", "out[o] = s + b[o];", "out[o] = s;"),
    ("per-word alpha from the first row only", "Sec. 4.1 (alpha of x)",
     "for (int t = 0; t < rows; ++t) {\n    float r = absmax", "for (int t = 0; t < 1; ++t) {\n    float r = absmax"),
]


def _compile(text: str, out: str) -> None:
    csrc = out[:-3] + ".c"
    with open(csrc, "w") as f:
        f.write(text)
    subprocess.check_call(["gcc", *O.GCC_FLAGS, csrc, "-o", out, "-lm"])


def _build_and_run_pins(job) -> subprocess.CompletedProcess:
    text, path = job
    _compile(text, path)
    env = dict(os.environ, AECCT_ORACLE_LIB=path)
    return subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider", "-m", "not gpu", *PINS],
                          cwd=ROOT, env=env, capture_output=True, text=True, timeout=900)


def test_each_planted_mistake_fails_a_pin(tmp_path):
    src = open(SRC).read()
    for name, _, old, new in MUTANTS:
        assert src.count(old) == 1, f"{name}: the original text must occur once"
        assert old != new
    names = ["unmodified"] + [m[0] for m in MUTANTS]
    texts = [src] + [src.replace(old, new) for _, _, old, new in MUTANTS]
    jobs = [(t, str(tmp_path / f"liboracle_{i}.so")) for i, t in enumerate(texts)]
    with ThreadPoolExecutor(max_workers=max(1, min(16, os.cpu_count() or 1))) as ex:
        results = list(ex.map(_build_and_run_pins, jobs))
    base = results[0]
    assert base.returncode == 0, "the unmodified oracle must pass its pins:\n" + base.stdout[-2000:]
    survivors, not_assertions = [], []
    for name, r in zip(names[1:], results[1:]):
        if r.returncode == 0:
            survivors.append(name)
        elif " failed" not in r.stdout.splitlines()[-1]:
            not_assertions.append(f"{name}: {r.stdout[-400:]}")
    assert not survivors, f"planted mistakes that no pin catches: {survivors}"
    assert not not_assertions, "mutants that stopped the pins without a failed assertion:\n" + "\n".join(not_assertions)
