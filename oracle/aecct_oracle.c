/*
 * AECCT inference forward pass -- CPU ORACLE.  TEST INFRASTRUCTURE ONLY.
 *
 * This file is the plain, slow reference that the CUDA decoder is checked against.
 * Only the test-suite, the smoke check and the CPU-baseline leg of the benchmark load
 * it.  It shares no code, header, table or constant with the CUDA library.
 *
 * It follows "Accelerating Error Correction Code Transformers" (Levy, Choukroun, Wolf):
 *   Sec. 3 (Problem Settings)       hard decision, syndrome, tokens h(y) = [|y|, 1-2s(y)]
 *   Sec. 3 (ECCT)                   per-position embedding, output head eps = W_o^T(W_{d->1} Phi)
 *   Sec. 4.1 eq. Ternary            AAP weight ternarisation (used by tests, not by decode)
 *   Sec. 4.1 eq. Quant              per-token absmax int8 activation quantisation
 *   Sec. 4.1 eq. AAPLinear          int accumulate, dequantise by gamma*delta*alpha/Q_b, add bias
 *   Sec. 3 (ECCT, linear_mode 1)    full-precision linear layers, on bf16 inputs and weights
 *   Sec. 4.2 (HPSA)                 first-ring heads on the c<->v mask, second-ring heads on the
 *                                   v<->v / c<->c mask
 *   Sec. 3 (ECCT, mask_mode 1)      the code-aware mask of the ECCT baseline: every head on the
 *                                   union of the two rings
 *   Sec. 4.3 eq. SPE                SPE table concatenated to the embedding (table given as input)
 *   Sec. 4 item 4                   ReLU in the feed-forward block (activation 0); GELU as the
 *                                   option activation 1 (x Phi(x), erf by Abramowitz & Stegun 7.1.26)
 *   Sec. 5 (Training & Inference)   Post-LN Transformer blocks
 *
 * Arithmetic is IEEE fp32 (the paper's FP32 model) with one canonical order of
 * operations wherever the paper leaves it open, so that any other implementation
 * of the same order reproduces these results bit for bit:
 *   - every multiply and add is rounded separately (build with -ffp-contract=off),
 *     except where fmaf() is written explicitly;
 *   - sums over a feature row use pairwise summation (recursive halving);
 *   - attention scores are taken in base-2 units: sigma = dot(q,k) * fp32(log2(e)/sqrt(d_h)),
 *     with dot(q,k) = (even-feature FMA chain) + (odd-feature FMA chain), each in feature order,
 *     p = 2^(sigma - max sigma), with 2^x evaluated by exp2_series() below (range
 *     reduction x = n + f, |f| <= 1/2, and the degree-7 Taylor series of e^(f ln 2));
 *   - sums over keys and over tokens run in ascending index order.
 *
 * Pins (tests/): exp2 against libm and its Taylor coefficients, GELU against the erf of libm and
 * its odd-part identity, pairwise sums, quantiser and
 * LayerNorm closed forms, brute-force integer products, masks against Tanner-graph distances,
 * codeword-symmetry invariance, the all-zero-weight closed form, and an independent float64
 * forward pass teacher-forced on the recorded integer core.  A planted-mistake test compiles
 * copies of this file with one mistake each and checks that every copy fails one of those pins.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORACLE_OK 0
#define ORACLE_EINVAL (-1)
#define ORACLE_ENOMEM (-3)

/* ------------------------------------------------------------------------- */
/* Model description (the oracle's own layout; unpacked int8 ternary weights) */
/* ------------------------------------------------------------------------- */
typedef struct {
  int32_t n, k, d, n_layers, heads, h_first, d_spe, ffn_mult, activation;
  int32_t mask_mode;       /* 0 = HPSA (Sec. 4.2); 1 = ECCT code-aware mask M1 | M2 for all heads (Sec. 3) */
  int32_t alpha_mode;      /* 0 = one alpha per token (C-1); 1 = one alpha per quantised matrix of a word */
  int32_t linear_mode;     /* 0 = AAP linears (Sec. 4.1); 1 = full-precision linears (ECCT, Sec. 3) on bf16 */
  const uint8_t *H;        /* [(n-k)][n] 0/1 */
  const float *emb;        /* [T][d-d_spe] */
  const float *spe;        /* [T][d_spe] */
  const int8_t *w;         /* per layer, in order q[d][d], k[d][d], v[d][d], o[d][d], ffn1[F][d], ffn2[d][F] */
  const float *w_scale;    /* [n_layers][6] */
  const float *bias;       /* per layer: bq[d] bk[d] bv[d] bo[d] b1[F] b2[d] */
  const float *ln_gamma;   /* [n_layers][2][d] */
  const float *ln_beta;    /* [n_layers][2][d] */
  const float *w_d1;       /* [d] */
  float b_d1;
  const float *w_out;      /* [T][n] */
  const float *b_out;      /* [n] */
  float ln_eps;
  float alpha_floor;
  const float *w_full;     /* linear_mode 1: fp32 weights, same order and shapes as w */
} oracle_model;

/* Optional record of the integer core for the first cap_B codewords.
 * gemm index g: 0 = QKV (K=d, N=3d), 1 = O (K=d, N=d), 2 = FFN1 (K=d, N=4d), 3 = FFN2 (K=4d, N=d).
 * q     int8  [cap_B][n_layers][4][T][4d]  quantised GEMM input (first K entries of a row used)
 * acc   int32 [cap_B][n_layers][4][T][4d]  integer accumulators (first N entries used); with
 *                                          linear_mode 1 the bit patterns of the fp32 sums, and
 *                                          q and alpha are left untouched
 * alpha fp32  [cap_B][n_layers][4][T]      max(absmax, floor) of the GEMM input row
 * syn   uint8 [cap_B][n-k]                 syndrome of the channel output */
typedef struct {
  int64_t cap_B;
  int8_t *q;
  int32_t *acc;
  float *alpha;
  uint8_t *syn;
} oracle_capture;

/* ------------------------------------------------------------------------- */
/* Canonical scalar pieces                                                   */
/* ------------------------------------------------------------------------- */

/* 2^x for x <= 0 (Sec. 4.2 softmax, canonical base-2 form).  Range reduction
 * x = n + f with n = rint(x), |f| <= 1/2, 2^f = e^(f ln2) = sum_k (f ln2)^k / k!
 * truncated after k = 7 and evaluated by Horner's rule with fused multiply-adds;
 * 2^n applied exactly with ldexpf.  Inputs below -125 give 0. */
static float g_exp2_coef[8];
__attribute__((constructor)) static void exp2_series_init(void) {
  double ln2 = 0.69314718055994530941723212145818;
  double term = 1.0;
  for (int k = 0; k < 8; ++k) {
    g_exp2_coef[k] = (float)term;
    term = term * ln2 / (double)(k + 1);
  }
}

float oracle_exp2_series(float x) {
  if (!(x >= -125.0f)) return 0.0f;
  float n = rintf(x);
  float f = x - n;
  float p = g_exp2_coef[7];
  for (int k = 6; k >= 0; --k) p = fmaf(p, f, g_exp2_coef[k]);
  return ldexpf(p, (int)n);
}

/* GELU(x) = x Phi(x) = 0.5 x (1 + erf(x / sqrt 2)) (activation 1).  erf by the rational
 * approximation 7.1.26 of Abramowitz & Stegun, Handbook of Mathematical Functions
 * (|error| <= 1.5e-7 for x >= 0, odd symmetry below 0), in fixed fp32 steps:
 *   z = x * fp32(1/sqrt 2), t = 1 / (1 + p |z|) (one fused multiply-add, then an IEEE divide),
 *   poly = t * (a1 + t (a2 + t (a3 + t (a4 + t a5)))) (Horner with fused multiply-adds, then a multiply),
 *   e = 2^((|z| * |z|) * fp32(-log2 e)) by exp2_series, erf|z| = 1 - poly * e,
 *   GELU = (0.5 x) * (1 + sign(z) erf|z|). */
float oracle_gelu(float x) {
  float z = x * 0.70710678118654752f;
  float az = fabsf(z);
  float t = 1.0f / fmaf(0.3275911f, az, 1.0f);
  float q = 1.061405429f;
  q = fmaf(q, t, -1.453152027f);
  q = fmaf(q, t, 1.421413741f);
  q = fmaf(q, t, -0.284496736f);
  q = fmaf(q, t, 0.254829592f);
  q = q * t;
  float e = oracle_exp2_series((az * az) * -1.44269504088896341f);
  float er = 1.0f - q * e;
  return (0.5f * x) * (1.0f + (z < 0.0f ? -er : er));
}

/* pairwise sum of v[0..len) (len a power of two): sum(lo half) + sum(hi half) */
float oracle_psum(const float *v, int len) {
  if (len == 1) return v[0];
  int h = len / 2;
  float a = oracle_psum(v, h);
  float b = oracle_psum(v + h, len - h);
  return a + b;
}

/* Sec. 3: bin(y) = 0.5(1 - sign(y)); y = 0 is read as a 0 bit. */
void oracle_hard_decision(const float *y, int n, uint8_t *b) {
  for (int j = 0; j < n; ++j) b[j] = (y[j] < 0.0f) ? 1 : 0;
}

/* Sec. 3: s = H b over GF(2). */
void oracle_syndrome(const uint8_t *H, int m, int n, const uint8_t *b, uint8_t *s) {
  for (int i = 0; i < m; ++i) {
    uint8_t acc = 0;
    for (int j = 0; j < n; ++j) acc ^= (uint8_t)(H[(size_t)i * n + j] & b[j]);
    s[i] = acc;
  }
}

/* Sec. 4.2 HPSA masks over the T = 2n-k Tanner-graph nodes (variables 0..n-1, checks n..T-1).
 * M1 (first ring): variable j <-> check i iff H_ij = 1 (no self loops).
 * M2 (second ring): variables j,j' that share a check; checks i,i' that share a variable;
 *                   a node with any neighbour is at distance 0 from itself and is kept. */
void oracle_masks(const uint8_t *H, int m, int n, uint8_t *M1, uint8_t *M2) {
  int T = n + m;
  memset(M1, 0, (size_t)T * T);
  memset(M2, 0, (size_t)T * T);
  for (int i = 0; i < m; ++i)
    for (int j = 0; j < n; ++j)
      if (H[(size_t)i * n + j]) {
        M1[(size_t)j * T + (n + i)] = 1;
        M1[(size_t)(n + i) * T + j] = 1;
      }
  for (int a = 0; a < n; ++a)
    for (int b = 0; b < n; ++b) {
      uint8_t hit = 0;
      for (int i = 0; i < m && !hit; ++i) hit = H[(size_t)i * n + a] & H[(size_t)i * n + b];
      M2[(size_t)a * T + b] = hit;
    }
  for (int a = 0; a < m; ++a)
    for (int b = 0; b < m; ++b) {
      uint8_t hit = 0;
      for (int j = 0; j < n && !hit; ++j) hit = H[(size_t)a * n + j] & H[(size_t)b * n + j];
      M2[(size_t)(n + a) * T + (n + b)] = hit;
    }
}

/* Sec. 4.1 eq. Quant, one token row: alpha = ||x||_inf, Q_b = 127,
 * q = RoundClip(x * (Q_b / alpha), -Q_b, Q_b), round half to even.
 * alpha is floored at alpha_floor so an all-zero row quantises to zeros. */
static float absmax(const float *x, int len) {
  float a = 0.0f;
  for (int i = 0; i < len; ++i) {
    float ax = fabsf(x[i]);
    if (ax > a) a = ax;
  }
  return a;
}
/* q = RoundClip(x * (Q_b / a), -Q_b, Q_b) for a given (floored) alpha a */
static void quant_with_alpha(const float *x, int len, float a, int8_t *q) {
  float r = 127.0f / a;
  for (int i = 0; i < len; ++i) {
    float v = rintf(x[i] * r);
    if (v > 127.0f) v = 127.0f;
    if (v < -127.0f) v = -127.0f;
    q[i] = (int8_t)v;
  }
}
void oracle_quant_row(const float *x, int len, float alpha_floor, int8_t *q, float *alpha_out) {
  float a = absmax(x, len);
  if (!(a > alpha_floor)) a = alpha_floor;
  quant_with_alpha(x, len, a, q);
  *alpha_out = a;
}
/* The alternative granularity (Sec. 4.1 writes alpha as a scalar of the whole input x in
 * R^{m x n}): alpha = ||x||_inf over all rows of a word's matrix, floored. */
static float matrix_alpha(const float *x, int rows, int len, size_t stride, float alpha_floor) {
  float a = 0.0f;
  for (int t = 0; t < rows; ++t) {
    float r = absmax(x + (size_t)t * stride, len);
    if (r > a) a = r;
  }
  if (!(a > alpha_floor)) a = alpha_floor;
  return a;
}

/* Sec. 4.1 eq. AAPLinear for one row: acc_o = sum_i q_i t_oi (exact integer), then
 * out_o = acc_o * (gamma*delta * alpha / Q_b) + b_o. */
void oracle_aap_linear_row(const int8_t *q, float alpha, int K, const int8_t *W, int N, float s_w,
                           const float *b, int32_t *acc_out, float *out) {
  float f = (s_w * alpha) / 127.0f;
  for (int o = 0; o < N; ++o) {
    int32_t acc = 0;
    const int8_t *wr = W + (size_t)o * K;
    for (int i = 0; i < K; ++i) acc += (int32_t)q[i] * (int32_t)wr[i];
    if (acc_out) acc_out[o] = acc;
    out[o] = (float)acc * f + b[o];
  }
}

/* bf16 value of a finite fp32 x, rounded to nearest even: keep the sign, the exponent and the top
 * 7 fraction bits; the 16 dropped bits round up when above half an ulp, or at exactly half when
 * the kept part is odd. */
float oracle_bf16_round(float x) {
  uint32_t u;
  memcpy(&u, &x, 4);
  uint32_t low = u & 0xFFFFu, keep = u & 0xFFFF0000u;
  if (low > 0x8000u || (low == 0x8000u && (keep & 0x10000u))) keep += 0x10000u;
  float r;
  memcpy(&r, &keep, 4);
  return r;
}

/* The full-precision linear layer of the ECCT baseline (Sec. 3) in the number format of the
 * tensor cores: out_o = fp32(sum_i bf16(x_i) bf16(W_oi)) + b_o.  Each product of two bf16 values
 * is exact in double and the sum runs in double (ascending i); it stays exact while the products
 * span fewer than 53 bits (always for the activations and weights here), so the sum is rounded
 * to fp32 once.  sum_out receives that fp32 sum (before the bias). */
void oracle_full_linear_row(const float *x, int K, const float *W, int N, const float *b, float *sum_out,
                            float *out) {
  double xb[4096];
  for (int i = 0; i < K; ++i) xb[i] = (double)oracle_bf16_round(x[i]);
  for (int o = 0; o < N; ++o) {
    const float *wr = W + (size_t)o * K;
    double acc = 0.0;
    for (int i = 0; i < K; ++i) acc += xb[i] * (double)oracle_bf16_round(wr[i]);
    float s = (float)acc;
    if (sum_out) sum_out[o] = s;
    out[o] = s + b[o];
  }
}

/* Sec. 4.1 eq. Ternary: gamma = Percentile(|W|, 0.5) (linear interpolation between order
 * statistics), t = RoundClip(W / (gamma*delta + eps), -1, 1); returns scale gamma*delta. */
static int cmp_float(const void *a, const void *b) {
  float x = *(const float *)a, y = *(const float *)b;
  return (x > y) - (x < y);
}
int oracle_ternary(const float *W, int64_t len, float delta, float eps, int8_t *t, float *scale_out) {
  if (len <= 0) return ORACLE_EINVAL;
  float *absw = (float *)malloc(sizeof(float) * (size_t)len);
  if (!absw) return ORACLE_ENOMEM;
  for (int64_t i = 0; i < len; ++i) absw[i] = fabsf(W[i]);
  qsort(absw, (size_t)len, sizeof(float), cmp_float);
  double pos = 0.5 * (double)(len - 1);
  int64_t lo = (int64_t)floor(pos);
  int64_t hi = lo + 1 < len ? lo + 1 : lo;
  double frac = pos - (double)lo;
  float gamma = (float)((double)absw[lo] + frac * ((double)absw[hi] - (double)absw[lo]));
  free(absw);
  float sc = gamma * delta;
  float den = sc + eps;
  for (int64_t i = 0; i < len; ++i) {
    float v = rintf(W[i] / den);
    if (v > 1.0f) v = 1.0f;
    if (v < -1.0f) v = -1.0f;
    t[i] = (int8_t)v;
  }
  *scale_out = sc;
  return ORACLE_OK;
}

/* LayerNorm of one row (Sec. 5 Post-LN): mu = psum(v)/d, var = psum((v-mu)^2)/d (biased),
 * y = ((v - mu) * (1/sqrt(var + eps))) * gamma + beta.  d is a power of two. */
void oracle_layernorm_row(const float *v, int d, const float *g, const float *b, float eps, float *y) {
  float tmp[1024];
  float inv_d = 1.0f / (float)d;
  float mu = oracle_psum(v, d) * inv_d;
  for (int i = 0; i < d; ++i) {
    float t = v[i] - mu;
    tmp[i] = t * t;
  }
  float var = oracle_psum(tmp, d) * inv_d;
  float rstd = 1.0f / sqrtf(var + eps);
  for (int i = 0; i < d; ++i) y[i] = ((v[i] - mu) * rstd) * g[i] + b[i];
}

/* Sec. 4.2 HPSA for one token set: Q,K,V,A are [T][d]; head e owns columns [e*dh, (e+1)*dh);
 * heads e < h_first attend over M1, the rest over M2.  Masked-out keys are skipped.
 * sigma_u = dot(Q_t, K_u) * c, c = fp32(log2(e)/sqrt(dh)); p_u = 2^(sigma_u - max);
 * A_t = (sum_u p_u V_u) * (1 / sum_u p_u).  A row with no key gets zeros. */
/* q . k over one head (Sec. 4.2): the even-indexed and the odd-indexed feature products each
 * summed by a chain of fused multiply-adds in feature order, then added (canonical order). */
static float oracle_dot(const float *q, const float *k, int dh) {
  float de = 0.0f, dod = 0.0f;
  for (int i = 0; i < dh; i += 2) {
    de = fmaf(q[i], k[i], de);
    dod = fmaf(q[i + 1], k[i + 1], dod);
  }
  return de + dod;
}

void oracle_attention(const float *Q, const float *K, const float *V, int T, int d, int heads,
                      int h_first, const uint8_t *M1, const uint8_t *M2, float *A) {
  int dh = d / heads;
  float c = (float)(1.4426950408889634074 / sqrt((double)dh));
  for (int t = 0; t < T; ++t) {
    for (int e = 0; e < heads; ++e) {
      const uint8_t *M = (e < h_first ? M1 : M2) + (size_t)t * T;
      const float *q = Q + (size_t)t * d + e * dh;
      float mx = -INFINITY;
      int any = 0;
      for (int u = 0; u < T; ++u) {
        if (!M[u]) continue;
        const float *kk = K + (size_t)u * d + e * dh;
        float s = oracle_dot(q, kk, dh) * c;
        if (!any || s > mx) mx = s;
        any = 1;
      }
      float *a = A + (size_t)t * d + e * dh;
      if (!any) {
        for (int i = 0; i < dh; ++i) a[i] = 0.0f;
        continue;
      }
      float l = 0.0f;
      float num[64];
      for (int i = 0; i < dh; ++i) num[i] = 0.0f;
      for (int u = 0; u < T; ++u) {
        if (!M[u]) continue;
        const float *kk = K + (size_t)u * d + e * dh;
        const float *vv = V + (size_t)u * d + e * dh;
        float p = oracle_exp2_series(oracle_dot(q, kk, dh) * c - mx);
        l = l + p;
        for (int i = 0; i < dh; ++i) num[i] = fmaf(p, vv[i], num[i]);
      }
      float inv = 1.0f / l;
      for (int i = 0; i < dh; ++i) a[i] = num[i] * inv;
    }
  }
}

/* ------------------------------------------------------------------------- */
/* Whole forward pass                                                        */
/* ------------------------------------------------------------------------- */
typedef struct {
  float *x, *qf, *kf, *vf, *a, *o, *u, *v, *z, *eps;
  int8_t *q;
  float *alpha;
  int32_t *acc;
  uint8_t *b, *s, *c;
  uint8_t *M1, *M2;
} work_t;

static int64_t cap_row_off(const oracle_model *m, int64_t bi, int l, int g, int t) {
  int T = 2 * m->n - m->k;
  int W4 = 4 * m->d;
  return ((((bi * m->n_layers + l) * 4 + g) * (int64_t)T) + t) * W4;
}

static void decode_one(const oracle_model *m, const float *y, uint8_t *bits, uint8_t *syn,
                       float *logits, work_t *w, const oracle_capture *cap, int64_t bi) {
  const int n = m->n, mm = m->n - m->k, T = 2 * m->n - m->k, d = m->d;
  const int F = m->ffn_mult * d, de = d - m->d_spe;
  const int capture = cap && cap->cap_B > bi;
  /* S1: hard decision and syndrome (Sec. 3) */
  oracle_hard_decision(y, n, w->b);
  oracle_syndrome(m->H, mm, n, w->b, w->s);
  if (capture && cap->syn) memcpy(cap->syn + bi * mm, w->s, (size_t)mm);
  /* S2: tokens h(y) = [|y|, 1 - 2 s], per-position embedding, SPE concatenation */
  for (int t = 0; t < T; ++t) {
    float h = t < n ? fabsf(y[t]) : 1.0f - 2.0f * (float)w->s[t - n];
    for (int c = 0; c < de; ++c) w->x[(size_t)t * d + c] = h * m->emb[(size_t)t * de + c];
    for (int c = 0; c < m->d_spe; ++c) w->x[(size_t)t * d + de + c] = m->spe[(size_t)t * m->d_spe + c];
  }
  size_t wlayer = (size_t)4 * d * d + (size_t)2 * F * d;
  size_t blayer = (size_t)5 * d + F;
  const int full = m->linear_mode == 1;
  for (int l = 0; l < m->n_layers; ++l) {
    const int8_t *Wq = full ? NULL : m->w + wlayer * l;
    const int8_t *Wk = full ? NULL : Wq + (size_t)d * d;
    const int8_t *Wv = full ? NULL : Wk + (size_t)d * d;
    const int8_t *Wo = full ? NULL : Wv + (size_t)d * d;
    const int8_t *W1 = full ? NULL : Wo + (size_t)d * d;
    const int8_t *W2 = full ? NULL : W1 + (size_t)F * d;
    /* full-precision weights, same order */
    const float *Fq = full ? m->w_full + wlayer * l : NULL;
    const float *Fk = full ? Fq + (size_t)d * d : NULL;
    const float *Fv = full ? Fk + (size_t)d * d : NULL;
    const float *Fo = full ? Fv + (size_t)d * d : NULL;
    const float *F1 = full ? Fo + (size_t)d * d : NULL;
    const float *F2 = full ? F1 + (size_t)F * d : NULL;
    const float *sw = full ? NULL : m->w_scale + (size_t)6 * l;
    const float *bq = m->bias + blayer * l, *bk = bq + d, *bv = bk + d, *bo = bv + d, *b1 = bo + d, *b2 = b1 + F;
    const float *g1 = m->ln_gamma + (size_t)2 * d * l, *g2 = g1 + d;
    const float *be1 = m->ln_beta + (size_t)2 * d * l, *be2 = be1 + d;
    const int per_word = m->alpha_mode == 1;
    /* S3/S4: Quant(x) and the Q, K, V AAP-linear layers (Sec. 4.1), or the full-precision ones */
    const float aw0 = per_word ? matrix_alpha(w->x, T, d, (size_t)d, m->alpha_floor) : 0.0f;
    for (int t = 0; t < T; ++t) {
      int8_t *qr = w->q + (size_t)t * F;
      float al = 0.0f;
      int32_t *ar = w->acc + (size_t)t * 3 * d;
      const float *xr = w->x + (size_t)t * d;
      if (full) {
        float *sr = (float *)ar;
        oracle_full_linear_row(xr, d, Fq, d, bq, sr, w->qf + (size_t)t * d);
        oracle_full_linear_row(xr, d, Fk, d, bk, sr + d, w->kf + (size_t)t * d);
        oracle_full_linear_row(xr, d, Fv, d, bv, sr + 2 * d, w->vf + (size_t)t * d);
      } else {
        if (per_word) quant_with_alpha(xr, d, al = aw0, qr);
        else oracle_quant_row(xr, d, m->alpha_floor, qr, &al);
        oracle_aap_linear_row(qr, al, d, Wq, d, sw[0], bq, ar, w->qf + (size_t)t * d);
        oracle_aap_linear_row(qr, al, d, Wk, d, sw[1], bk, ar + d, w->kf + (size_t)t * d);
        oracle_aap_linear_row(qr, al, d, Wv, d, sw[2], bv, ar + 2 * d, w->vf + (size_t)t * d);
      }
      if (capture) {
        int64_t off = cap_row_off(m, bi, l, 0, t);
        if (cap->q && !full) memcpy(cap->q + off, qr, (size_t)d);
        if (cap->acc) memcpy(cap->acc + off, ar, sizeof(int32_t) * 3 * d);
        if (cap->alpha && !full) cap->alpha[off / (4 * d)] = al;
      }
    }
    /* S5: HPSA (Sec. 4.2) */
    oracle_attention(w->qf, w->kf, w->vf, T, d, m->heads, m->h_first, w->M1, w->M2, w->a);
    /* S6: O projection, residual, LayerNorm (Post-LN, Sec. 5) */
    const float aw1 = per_word ? matrix_alpha(w->a, T, d, (size_t)d, m->alpha_floor) : 0.0f;
    for (int t = 0; t < T; ++t) {
      int8_t *qr = w->q + (size_t)t * F;
      float al = 0.0f;
      int32_t *ar = w->acc + (size_t)t * 4 * d;
      const float *arow = w->a + (size_t)t * d;
      if (full) {
        oracle_full_linear_row(arow, d, Fo, d, bo, (float *)ar, w->o + (size_t)t * d);
      } else {
        if (per_word) quant_with_alpha(arow, d, al = aw1, qr);
        else oracle_quant_row(arow, d, m->alpha_floor, qr, &al);
        oracle_aap_linear_row(qr, al, d, Wo, d, sw[3], bo, ar, w->o + (size_t)t * d);
      }
      for (int c = 0; c < d; ++c) w->v[c] = w->x[(size_t)t * d + c] + w->o[(size_t)t * d + c];
      oracle_layernorm_row(w->v, d, g1, be1, m->ln_eps, w->x + (size_t)t * d);
      if (capture) {
        int64_t off = cap_row_off(m, bi, l, 1, t);
        if (cap->q && !full) memcpy(cap->q + off, qr, (size_t)d);
        if (cap->acc) memcpy(cap->acc + off, ar, sizeof(int32_t) * d);
        if (cap->alpha && !full) cap->alpha[off / (4 * d)] = al;
      }
    }
    /* S7/S8: FFN with ReLU (Sec. 4 item 4) or GELU, residual, LayerNorm */
    const float aw2 = per_word ? matrix_alpha(w->x, T, d, (size_t)d, m->alpha_floor) : 0.0f;
    for (int t = 0; t < T; ++t) {
      int8_t *qr = w->q + (size_t)t * F;
      float al = 0.0f;
      int32_t *ar = w->acc + (size_t)t * 4 * d;
      float *ur = w->u + (size_t)t * F;
      const float *xr = w->x + (size_t)t * d;
      if (full) {
        oracle_full_linear_row(xr, d, F1, F, b1, (float *)ar, ur);
      } else {
        if (per_word) quant_with_alpha(xr, d, al = aw2, qr);
        else oracle_quant_row(xr, d, m->alpha_floor, qr, &al);
        oracle_aap_linear_row(qr, al, d, W1, F, sw[4], b1, ar, ur);
      }
      if (capture) {
        int64_t off = cap_row_off(m, bi, l, 2, t);
        if (cap->q && !full) memcpy(cap->q + off, qr, (size_t)d);
        if (cap->acc) memcpy(cap->acc + off, ar, sizeof(int32_t) * F);
        if (cap->alpha && !full) cap->alpha[off / (4 * d)] = al;
      }
      if (m->activation == 0)
        for (int c = 0; c < F; ++c) ur[c] = ur[c] > 0.0f ? ur[c] : 0.0f;
      else
        for (int c = 0; c < F; ++c) ur[c] = oracle_gelu(ur[c]);
    }
    const float aw3 = per_word ? matrix_alpha(w->u, T, F, (size_t)F, m->alpha_floor) : 0.0f;
    for (int t = 0; t < T; ++t) {
      int8_t *qr = w->q + (size_t)t * F;
      float al = 0.0f;
      int32_t *ar = w->acc + (size_t)t * 4 * d;
      const float *ur = w->u + (size_t)t * F;
      if (full) {
        oracle_full_linear_row(ur, F, F2, d, b2, (float *)ar, w->o);
      } else {
        if (per_word) quant_with_alpha(ur, F, al = aw3, qr);
        else oracle_quant_row(ur, F, m->alpha_floor, qr, &al);
        oracle_aap_linear_row(qr, al, F, W2, d, sw[5], b2, ar, w->o);
      }
      for (int c = 0; c < d; ++c) w->v[c] = w->x[(size_t)t * d + c] + w->o[c];
      oracle_layernorm_row(w->v, d, g2, be2, m->ln_eps, w->x + (size_t)t * d);
      if (capture) {
        int64_t off = cap_row_off(m, bi, l, 3, t);
        if (cap->q && !full) memcpy(cap->q + off, qr, (size_t)F);
        if (cap->acc) memcpy(cap->acc + off, ar, sizeof(int32_t) * d);
        if (cap->alpha && !full) cap->alpha[off / (4 * d)] = al;
      }
    }
  }
  /* S9: output head eps = W_o^T (W_{d->1} Phi) + biases (Sec. 3) */
  for (int t = 0; t < T; ++t) {
    for (int c = 0; c < d; ++c) w->v[c] = w->x[(size_t)t * d + c] * m->w_d1[c];
    w->z[t] = oracle_psum(w->v, d) + m->b_d1;
  }
  for (int j = 0; j < n; ++j) {
    float e = 0.0f;
    for (int t = 0; t < T; ++t) e = fmaf(m->w_out[(size_t)t * n + j], w->z[t], e);
    w->eps[j] = e + m->b_out[j];
  }
  /* S10: x_hat = y * eps; decoded bit = [x_hat < 0]; syndrome of the decoded word */
  for (int j = 0; j < n; ++j) {
    w->c[j] = (y[j] * w->eps[j] < 0.0f) ? 1 : 0;
    if (bits) bits[j] = w->c[j];
    if (logits) logits[j] = w->eps[j];
  }
  if (syn) oracle_syndrome(m->H, mm, n, w->c, syn);
}

static int work_alloc(const oracle_model *m, work_t *w) {
  int T = 2 * m->n - m->k, d = m->d, F = m->ffn_mult * d;
  memset(w, 0, sizeof(*w));
  w->x = (float *)calloc((size_t)T * d, sizeof(float));
  w->qf = (float *)calloc((size_t)T * d, sizeof(float));
  w->kf = (float *)calloc((size_t)T * d, sizeof(float));
  w->vf = (float *)calloc((size_t)T * d, sizeof(float));
  w->a = (float *)calloc((size_t)T * d, sizeof(float));
  w->o = (float *)calloc((size_t)T * d, sizeof(float));
  w->u = (float *)calloc((size_t)T * F, sizeof(float));
  w->v = (float *)calloc((size_t)(d > T ? d : T), sizeof(float));
  w->z = (float *)calloc((size_t)T, sizeof(float));
  w->eps = (float *)calloc((size_t)m->n, sizeof(float));
  w->q = (int8_t *)calloc((size_t)T * F, 1);
  w->acc = (int32_t *)calloc((size_t)T * F, sizeof(int32_t));
  w->b = (uint8_t *)calloc((size_t)m->n, 1);
  w->s = (uint8_t *)calloc((size_t)m->n, 1);
  w->c = (uint8_t *)calloc((size_t)m->n, 1);
  w->M1 = (uint8_t *)calloc((size_t)T * T, 1);
  w->M2 = (uint8_t *)calloc((size_t)T * T, 1);
  if (!w->x || !w->qf || !w->kf || !w->vf || !w->a || !w->o || !w->u || !w->v || !w->z || !w->eps ||
      !w->q || !w->acc || !w->b || !w->s || !w->c || !w->M1 || !w->M2)
    return ORACLE_ENOMEM;
  oracle_masks(m->H, m->n - m->k, m->n, w->M1, w->M2);
  if (m->mask_mode == 1) {
    /* ECCT's code-aware mask (Sec. 3): a token attends to its Tanner neighbours, to the nodes of
     * its own type two edges away, and to itself -- the union of the two rings -- in every head */
    const size_t TT = (size_t)(2 * m->n - m->k) * (size_t)(2 * m->n - m->k);
    for (size_t i = 0; i < TT; ++i) w->M1[i] = w->M2[i] = (uint8_t)(w->M1[i] | w->M2[i]);
  }
  return ORACLE_OK;
}

static void work_free(work_t *w) {
  free(w->x); free(w->qf); free(w->kf); free(w->vf); free(w->a); free(w->o); free(w->u);
  free(w->v); free(w->z); free(w->eps); free(w->q); free(w->acc); free(w->b); free(w->s);
  free(w->c); free(w->M1); free(w->M2);
}

typedef struct {
  const oracle_model *m;
  const float *y;
  uint8_t *bits, *syn;
  float *logits;
  const oracle_capture *cap;
  int64_t b0, b1;
  int rc;
} job_t;

static void *run_job(void *arg) {
  job_t *j = (job_t *)arg;
  work_t w;
  j->rc = work_alloc(j->m, &w);
  if (j->rc == ORACLE_OK) {
    int n = j->m->n, mm = j->m->n - j->m->k;
    for (int64_t b = j->b0; b < j->b1; ++b)
      decode_one(j->m, j->y + b * n, j->bits ? j->bits + b * n : NULL, j->syn ? j->syn + b * mm : NULL,
                 j->logits ? j->logits + b * n : NULL, &w, j->cap, b);
  }
  work_free(&w);
  return NULL;
}

static int validate(const oracle_model *m) {
  if (!m || !m->H || !m->emb || !m->w || !m->w_scale || !m->bias || !m->ln_gamma || !m->ln_beta ||
      !m->w_d1 || !m->w_out || !m->b_out)
    return ORACLE_EINVAL;
  if (m->n <= 0 || m->k <= 0 || m->k >= m->n || m->d <= 0 || m->heads <= 0 || m->d % m->heads) return ORACLE_EINVAL;
  if (m->d & (m->d - 1)) return ORACLE_EINVAL; /* pairwise LN sums take a power-of-two width */
  if (m->d > 1024 || m->d / m->heads > 64 || (m->d / m->heads) % 2 || m->n_layers < 0) return ORACLE_EINVAL;
  if (m->h_first < 0 || m->h_first > m->heads || m->d_spe < 0 || m->d_spe >= m->d) return ORACLE_EINVAL;
  if (m->mask_mode < 0 || m->mask_mode > 1 || m->alpha_mode < 0 || m->alpha_mode > 1) return ORACLE_EINVAL;
  if (m->linear_mode < 0 || m->linear_mode > 1) return ORACLE_EINVAL;
  if (m->linear_mode == 1 && (!m->w_full || m->alpha_mode != 0)) return ORACLE_EINVAL;
  if (m->d_spe > 0 && !m->spe) return ORACLE_EINVAL;
  if (m->ffn_mult != 4 || m->activation < 0 || m->activation > 1) return ORACLE_EINVAL; /* FFN width 4d, ReLU/GELU */
  return ORACLE_OK;
}

/* Decode B received words y[B][n] on nthreads host threads (contiguous split). */
int oracle_decode(const oracle_model *m, const float *y, int64_t B, uint8_t *bits, uint8_t *syn,
                  float *logits, int nthreads, const oracle_capture *cap) {
  exp2_series_init();
  int rc = validate(m);
  if (rc) return rc;
  if (B < 0 || (B > 0 && !y)) return ORACLE_EINVAL;
  if (B == 0) return ORACLE_OK;
  if (nthreads < 1) nthreads = 1;
  if (nthreads > B) nthreads = (int)B;
  job_t *jobs = (job_t *)calloc((size_t)nthreads, sizeof(job_t));
  pthread_t *th = (pthread_t *)calloc((size_t)nthreads, sizeof(pthread_t));
  if (!jobs || !th) {
    free(jobs); free(th);
    return ORACLE_ENOMEM;
  }
  for (int i = 0; i < nthreads; ++i) {
    jobs[i] = (job_t){m, y, bits, syn, logits, cap, B * i / nthreads, B * (i + 1) / nthreads, 0};
    if (nthreads == 1) run_job(&jobs[i]);
    else pthread_create(&th[i], NULL, run_job, &jobs[i]);
  }
  if (nthreads > 1)
    for (int i = 0; i < nthreads; ++i) pthread_join(th[i], NULL);
  rc = ORACLE_OK;
  for (int i = 0; i < nthreads; ++i)
    if (jobs[i].rc) rc = jobs[i].rc;
  free(jobs);
  free(th);
  return rc;
}

/* exposes the series coefficients for the tests (they must equal fp32(ln2^k / k!)) */
void oracle_exp2_coefficients(float *out8) {
  exp2_series_init();
  for (int k = 0; k < 8; ++k) out8[k] = g_exp2_coef[k];
}
