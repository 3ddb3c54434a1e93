/*
 * aecct.h -- C ABI of the GB300 (sm_103a) AECCT decoder library (libaecct.so).
 *
 * The library runs the batched inference forward pass of the Accelerated Error
 * Correction Code Transformer ("Accelerating Error Correction Code Transformers",
 * Levy, Choukroun, Wolf): received words y (Sec. 3, "Problem Settings") go through
 * the preprocessing h(y) = [|y|, 1 - 2 s(y)], a per-position embedding with the
 * spectral positional encoding concatenated (Sec. 4.3), N Post-LN encoder blocks
 * (Sec. 5) whose linear layers are AAP ternary-weight / int8-activation layers
 * (Sec. 4.1, eqs. Quant and AAPLinear) and whose attention is head-partitioned
 * (Sec. 4.2, HPSA), and the output head eps = W_o^T (W_{d->1} Phi) (Sec. 3, ECCT),
 * followed by hard decisions x_hat = y * eps (Sec. 3).
 *
 * Conventions
 *   - Every function returns an aecct_status (0 = success, negative = error).
 *   - Pointers documented as HOST are read during the call only; the caller keeps
 *     ownership.  Pointers documented as DEVICE must point to CUDA device memory of
 *     the current device; the caller keeps ownership.
 *   - The arithmetic is IEEE fp32 with one fixed order of operations (pairwise
 *     feature-row sums, separately rounded multiply/add in the quantiser and
 *     dequantiser, base-2 softmax with a degree-7 Taylor-series exp2, ascending key
 *     order), so results are deterministic and do not depend on the batch size or
 *     on how codewords are spread over the GPU.
 *   - A handle serves one decode at a time; concurrent decodes need separate handles.
 */
#ifndef AECCT_H
#define AECCT_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  AECCT_OK = 0,
  AECCT_ERR_INVALID_ARG = -1,  /* a dimension, value or pointer argument is invalid */
  AECCT_ERR_UNSUPPORTED = -2,  /* valid model outside the compiled kernel set (d, heads, T) */
  AECCT_ERR_OUT_OF_MEMORY = -3,
  AECCT_ERR_CUDA = -4,         /* a CUDA runtime call or kernel launch failed (see aecct_last_error) */
  AECCT_ERR_TIMEOUT = -5,      /* a device-side wait exceeded its limit; the kernel stopped early */
  AECCT_ERR_NO_DEVICE = -6     /* no sm_103 device is current */
} aecct_status;

typedef struct aecct_handle aecct_handle; /* opaque */

/*
 * Model description (inference form).  All pointers are HOST and are deep-copied by
 * aecct_create.  T = 2n - k tokens (n variable nodes, then n-k check nodes), F = 4d.
 *
 *   n, k          code length and dimension (0 < k < n); H has n-k rows.
 *   d             embedding width; this build supports d in {32, 64, 128}.
 *   n_layers      N >= 1 encoder blocks.
 *   heads         attention heads; this build supports heads == 8 (d_h = d/8).
 *   h_first       number of first-ring heads (Sec. 4.2); heads [0, h_first) attend over
 *                 the first-ring mask, heads [h_first, heads) over the second-ring mask.
 *   d_spe         width of the SPE table (0 <= d_spe < d); the per-position embedding
 *                 fills the first d - d_spe features (Sec. 4.3; Sec. 5 ablation text).
 *   ffn_mult      feed-forward width multiplier; must be 4.
 *   activation    0 = ReLU (Sec. 4 item 4); 1 = GELU, x Phi(x) = 0.5 x (1 + erf(x / sqrt 2)),
 *                 with erf by the rational approximation 7.1.26 of Abramowitz & Stegun
 *                 (|error| <= 1.5e-7) in a fixed fp32 order.  Other values are rejected.
 *   cluster_ctas  0 = choose automatically; otherwise the number of CTAs (1..8) that
 *                 share one group of codewords (tuning knob).
 *   attention_mode 0 = choose automatically; 1 = per-row neighbour lists (any cluster size);
 *                 2 = warp tasks over shared key sets (one CTA per group; d <= 64 with at most
 *                 128 tokens, or d = 128 with alpha_mode 0 and at most 128 rows once the checks'
 *                 rows start on the first 32-row boundary after the variables);
 *                 3 = per-row neighbour lists over per-head staged rows (d = 128, at most 640
 *                 token rows per group and 256 keys per row): head by head, the group's K and V
 *                 rows are gathered from every CTA of the cluster into local shared memory, and
 *                 the 4 threads of a row share its keys.  The default for d = 128 when a group
 *                 spans more than one CTA.  Every mode computes the same results bit for bit.
 *   mask_mode     0 = HPSA (Sec. 4.2): heads [0, h_first) first ring, the rest second ring;
 *                 1 = the ECCT code-aware mask (Sec. 3) for every head: the union of the first
 *                 and second rings (which contains each node itself).  Other values are rejected.
 *   alpha_mode    absmax granularity of eq. Quant (Sec. 4.1): 0 = one alpha per token row;
 *                 1 = one alpha per quantised matrix of a codeword (the max over its T rows).
 *                 1 needs one CTA per codeword (T <= 128 and cluster_ctas 0 or 1), else
 *                 AECCT_ERR_UNSUPPORTED.
 *   linear_mode   0 = AAP linear layers (Sec. 4.1): ternary w_packed, scales w_scale, int8
 *                 activations (eq. Quant, eq. AAPLinear).
 *                 1 = full-precision linear layers, as in the ECCT baseline (Sec. 3): weights
 *                 w_full (fp32, rounded once to bf16, round to nearest even), each GEMM input
 *                 row rounded to bf16 (round to nearest even), products accumulated in fp32 on
 *                 the tensor cores (order of the accumulation not specified), out = acc + b.
 *                 w_packed and w_scale are not read (may be NULL); alpha_mode must be 0.
 *   H             [(n-k)][n] uint8 row-major, entries 0/1, no all-zero row or column.
 *   emb           [T][d-d_spe] fp32: token t's embedding row, scaled by h_t (Sec. 3, ECCT).
 *   spe           [T][d_spe] fp32: spectral positional encoding table (Sec. 4.3);
 *                 may be NULL when d_spe == 0.
 *   w_packed      ternary weights of all blocks, 2 bits each.  Per block, in this order:
 *                 W_q [d][d], W_k [d][d], W_v [d][d], W_o [d][d], W_1 [F][d], W_2 [d][F]
 *                 (row = output unit, d_out rows of d_in weights).  A row of d_in weights
 *                 takes d_in/4 bytes; weight i sits in bits 2*(i%4)..2*(i%4)+1 of byte i/4,
 *                 coded 00 = 0, 01 = +1, 11 = -1 (10 is invalid).  Total bytes:
 *                 n_layers * 12 * d * d / 4.
 *   w_scale       [n_layers][6] per-tensor scales gamma*delta (eq. Ternary), same order.
 *   bias          per block d_q, d_k, d_v, d_o, F, d fp32 values (b_q b_k b_v b_o b_1 b_2).
 *   ln_gamma      [n_layers][2][d] LayerNorm weights (after attention, after FFN).
 *   ln_beta       [n_layers][2][d] LayerNorm biases.
 *   w_d1, b_d1    [d] and scalar: the W_{d->1} projection and its bias.
 *   w_out, b_out  [T][n] row-major and [n]: the W_o projection (T -> n) and its bias.
 *   ln_eps        LayerNorm epsilon (added to the biased variance).
 *   alpha_floor   lower bound on the absmax alpha of eq. Quant (an all-zero row maps to
 *                 zero codes instead of dividing by zero).
 *   wait_limit_cycles  0 = default (about 2^32 SM cycles); bound on every device-side
 *                 wait, after which the kernel stops and decode reports AECCT_ERR_TIMEOUT.
 *   w_full        linear_mode 1 only: fp32 weights of all blocks, per block W_q [d][d],
 *                 W_k [d][d], W_v [d][d], W_o [d][d], W_1 [F][d], W_2 [d][F] (row = output
 *                 unit), n_layers * 12 * d * d floats.  NULL when linear_mode is 0.
 */
typedef struct {
  int32_t n, k, d, n_layers, heads, h_first, d_spe, ffn_mult, activation, cluster_ctas, attention_mode, mask_mode;
  int32_t alpha_mode;
  int32_t linear_mode;
  const uint8_t *H;
  const float *emb;
  const float *spe;
  const uint8_t *w_packed;
  const float *w_scale;
  const float *bias;
  const float *ln_gamma;
  const float *ln_beta;
  const float *w_d1;
  float b_d1;
  const float *w_out;
  const float *b_out;
  float ln_eps;
  float alpha_floor;
  int64_t wait_limit_cycles;
  const float *w_full;
} aecct_model_desc;

/* Validate the description, build the HPSA masks from H (Sec. 4.2: first ring = Tanner
 * graph neighbours, second ring = nodes at distance two, plus the node itself), lay the
 * weights out for the tensor cores and copy everything to the current device (AAP linears:
 * the 2-bit codes are copied as they are and expanded into bf16 tensor-core tiles by a kernel
 * on the device; the call waits for it).  On
 * success *out receives a new handle.  Errors: INVALID_ARG (bad dimension, H not 0/1,
 * zero row/column in H, h_first > heads, d_spe >= d, packed code 10, NULL pointer),
 * UNSUPPORTED (d, heads, ffn_mult or T outside this build), NO_DEVICE, OUT_OF_MEMORY, CUDA. */
int aecct_create(const aecct_model_desc *desc, aecct_handle **out);

/* Decode B received words.  y_dev: DEVICE fp32 [B][n] channel outputs y = x_s + noise
 * (Sec. 3).  Outputs (DEVICE, written for every word):
 *   bits_dev      uint8 [B][n]: decoded bits, 1 where y_j * eps_j < 0 (x_hat = y * eps);
 *   syndrome_dev  uint8 [B][n-k] or NULL: H times the decoded bits over GF(2)
 *                 (all zero iff the decoded word is a codeword);
 *   logits_dev    fp32 [B][n] or NULL: the network output eps (multiplicative-noise
 *                 prediction, Sec. 3).
 * Runs asynchronously on cuda_stream (a cudaStream_t; NULL = legacy default stream).
 * B == 0 is a no-op.  y is expected finite: a NaN or infinity is not checked, and the words
 * it reaches get unspecified bits and logits (no value steers a memory access, so the
 * other words of the batch are unaffected).  Errors: INVALID_ARG (B < 0, NULL y/bits with
 * B > 0, or a current device other than the one the handle was created on), CUDA, and
 * TIMEOUT reported for an earlier decode on this handle whose kernel stopped. */
int aecct_decode(aecct_handle *h, const float *y_dev, int64_t B, uint8_t *bits_dev, uint8_t *syndrome_dev,
                 float *logits_dev, void *cuda_stream);

/* Same as aecct_decode but with HOST buffers (pageable or pinned): copies y to the device,
 * decodes, copies the outputs back and waits for completion.  Staging memory is owned by
 * the handle and grows on demand. */
int aecct_decode_host(aecct_handle *h, const float *y_host, int64_t B, uint8_t *bits_host, uint8_t *syndrome_host,
                      float *logits_host, void *cuda_stream);

/* The paper has no counterpart of this call (it is an implementation convenience).
 * The same decode as aecct_decode_host, with HOST buffers, that allocates nothing: the device
 * staging of y, bits, syndromes and logits and the kernel's status word live in one file-scope
 * static device array of AECCT_NOALLOC_SCRATCH_BYTES (4 MiB).  It serves callers that must not
 * allocate device memory while they decode: a process whose device memory is a fixed budget
 * taken up front, or a latency-bound loop in which a cudaMalloc/cudaFree (which may synchronise
 * the device) would stall other work.  aecct_decode_host instead grows its staging with
 * cudaMalloc.
 *   Limit: B words need B*(4n + n) bytes, + B*(n-k) with a syndrome, + B*4n with logits, each
 *   part rounded up to 256 bytes, plus 256 bytes for the status word, at most 4 MiB (Polar(64,32)
 *   with all outputs: 6,897 words).  A larger B returns AECCT_ERR_INVALID_ARG and
 *   aecct_last_error says so.
 *   Set-up: the first call on a device (that device current) resolves the array's address with
 *   cudaGetSymbolAddress; make that first call before any stream capture.
 *   Zeroing: the status word is cleared (cudaMemsetAsync on `cuda_stream`) before each launch;
 *   the staging needs no clearing (y is copied in, every output element is written).
 *   Concurrency: every call uses the same array, so calls that overlap in time (two host threads,
 *   or two streams whose work interleaves on the device) race; serialise them.
 *   Device: the current device must be the one the handle was created on (the array used is the
 *   current device's), else AECCT_ERR_INVALID_ARG.
 * An earlier asynchronous aecct_decode on the handle reports its status first, as in aecct_decode.
 * The call waits for its stream and returns the decode status (AECCT_ERR_TIMEOUT as
 * aecct_synchronize reports it). */
#define AECCT_NOALLOC_SCRATCH_BYTES (4u << 20)
int aecct_decode_host_noalloc(aecct_handle *h, const float *y_host, int64_t B, uint8_t *bits_host,
                              uint8_t *syndrome_host, float *logits_host, void *cuda_stream);

/* The AAP weight quantiser of Sec. 4.1 (eq. Ternary), as the training forward applies it to each
 * weight tensor (biases excluded), on the GPU:
 *   gamma = Percentile(|W|, 0.5): the median of |W|, interpolated linearly between the two middle
 *     order statistics (position 0.5 (len - 1)) when len is even;
 *   scale = gamma * delta (fp32);
 *   Ternary(W) = RoundClip(W / (scale + eps), -1, 1), an IEEE fp32 division, round to nearest even.
 * The straight-through estimator of training passes the gradient of scale * Ternary(W) to W
 * unchanged, so the forward values are all it needs.
 *   w_dev       DEVICE fp32, the n_tensors tensors back to back (tensor j has len_host[j]
 *               elements, a multiple of 4, at least 4, at most 2^31; finite values).
 *   len_host    HOST [n_tensors]; delta_host HOST [n_tensors] (the learnable delta, > 0).
 *   eps         > 0 (keeps the division finite when gamma delta is 0).
 *   packed_dev  DEVICE, len/4 bytes per tensor back to back: the 2-bit format of w_packed above
 *               (weight i of the tensor at bits 2 (i % 4) of byte i / 4: 00 = 0, 01 = +1, 11 = -1).
 *   scale_dev   DEVICE fp32 [n_tensors]: gamma * delta (the w_scale of aecct_create).
 *   wq_dev      DEVICE fp32 like w_dev, or NULL: scale * Ternary(W), the weights the training
 *               forward multiplies with.
 * Asynchronous on cuda_stream.  Errors: INVALID_ARG (a length or delta out of range, eps <= 0,
 * a NULL pointer), CUDA. */
int aecct_aap_ternarize(const float *w_dev, int32_t n_tensors, const int64_t *len_host, const float *delta_host,
                        float eps, uint8_t *packed_dev, float *scale_dev, float *wq_dev, void *cuda_stream);

/* The spectral positional encoding of Sec. 4.3 computed on the GPU, in double precision: the table
 * aecct_create takes as `spe`.  Tanner graph of H (variables 0..n-1, checks n..n+m-1, m = n - k,
 * T = n + m <= 1024 nodes), Laplacian L = D - A, its eigenpairs (lambda_i, phi_i) in ascending order
 * (parallel Jacobi rotations) in the canonical basis (per cluster of eigenvalues within 1e-8 max(1,
 * |lambda|max) of each other: Gram-Schmidt of P e_0, P e_1, ... in node order, P the cluster's
 * projector, residuals of norm <= 1e-6 skipped; a simple eigenvalue's vector has a positive first
 * entry above 1e-6 in magnitude), then for every node j:
 *   X_j = Phi_j W_pe, Phi_j row i = (lambda_i, phi_i[j]);
 *   MHSA(X_j) = [softmax((X_j Wq_e)(X_j Wk_e)^T / sqrt(d_e)) (X_j Wv_e)]_e Wo, d_e = d_spe / heads;
 *   SPE_j = the mean of the T rows of MHSA(X_j) (average pooling as the reduction W_{(2n-k)->1}).
 * All pointers HOST: H [(n-k)][n] 0/1; w_pe [2][d_spe]; wq, wk, wv [heads][d_spe][d_e]; wo
 * [d_spe][d_spe] (fp64, row-major).  Outputs: spe_out fp32 [T][d_spe]; lam_out [T], U_out [T][T]
 * (column i = eigenvector i), spe64_out [T][d_spe] fp64, each NULL when not wanted.  Synchronous;
 * allocates and frees its device memory.  Errors: INVALID_ARG, UNSUPPORTED (a cluster's basis came
 * out short), CUDA. */
int aecct_spe_table(const uint8_t *H, int32_t n, int32_t k, int32_t d_spe, int32_t heads, const double *w_pe,
                    const double *wq, const double *wk, const double *wv, const double *wo, float *spe_out,
                    double *lam_out, double *U_out, double *spe64_out);

/* Wait for the handle's last decode and report whether its kernel stopped on a
 * device-side timeout (AECCT_ERR_TIMEOUT) or a CUDA error occurred. */
int aecct_synchronize(aecct_handle *h);

/* Record the integer core of the next decodes for words 0..cap_B-1 (cap_B = 0 stops).
 * DEVICE buffers, caller-owned, T = 2n-k, W = 4d, gemm g: 0 = QKV (K = d, N = 3d,
 * columns q|k|v), 1 = O (K = d, N = d), 2 = FFN1 (K = d, N = 4d), 3 = FFN2 (K = 4d, N = d):
 *   q_dev      int8  [cap_B][n_layers][4][T][W]  Quant(x) codes of the GEMM input row (first K used)
 *   acc_dev    int32 [cap_B][n_layers][4][T][W]  integer accumulators sum_i q_i t_oi (first N used)
 *   alpha_dev  fp32  [cap_B][n_layers][4][T]     max(absmax, alpha_floor) of the input row
 *   syn_dev    uint8 [cap_B][n-k]                syndrome s(y) of the channel output (Sec. 3)
 * With full-precision linears (linear_mode 1) acc_dev receives the bit patterns of the fp32
 * accumulators, and q_dev and alpha_dev are not written.
 * Any of the four may be NULL.  Unused entries are left untouched. */
int aecct_set_capture(aecct_handle *h, int64_t cap_B, int8_t *q_dev, int32_t *acc_dev, float *alpha_dev,
                      uint8_t *syn_dev);

/* Launch facts of the handle (for benchmarks): CTAs per codeword group, codewords per
 * group, the number of clusters a decode launches at most, threads per CTA, dynamic
 * shared memory bytes per CTA (warp tasks: with their plan), and the attention mode in use (1 = per-row lists,
 * 2 = warp tasks, 3 = per-row lists over per-head staged rows).  Any pointer may be NULL. */
int aecct_query(const aecct_handle *h, int32_t *cluster_ctas, int32_t *words_per_group, int32_t *max_clusters,
                int32_t *threads_per_cta, int32_t *smem_bytes, int32_t *attention_mode);

int aecct_destroy(aecct_handle *h);

/* Static description of a status code. */
const char *aecct_status_string(int status);

/* Text of the last CUDA error seen by this thread inside the library ("" if none). */
const char *aecct_last_error(void);

/*
 * Diagnostics (no counterpart in the paper).
 *
 * aecct_selftest_mma: one CTA stages A [128][K] and B [N][K] (HOST int8 values, row-major,
 * converted to bf16) in shared memory, multiplies them on the tensor cores
 * (tcgen05.mma kind::f16, fp32 accumulators in tensor memory) and returns
 * out_host [128][N] fp32 = A * B^T.  K in {16, 32, ..., 128}, N in {16, 32, ..., 256}.
 *
 * aecct_selftest_timeout: one warp waits on a shared-memory barrier that nothing
 * completes, with a limit of limit_cycles; *status_host receives AECCT_ERR_TIMEOUT
 * when the bounded wait gave up as designed (AECCT_OK would mean the barrier completed).
 */
int aecct_selftest_mma(const int8_t *a_host, const int8_t *b_host, int32_t K, int32_t N, float *out_host);
int aecct_selftest_timeout(int64_t limit_cycles, int32_t *status_host);

/* aecct_selftest_fma_rate: the measured fp32 fused multiply-add rate of the current device, the
 * denominator of the CUDA-core roofline that the benchmark reports.  A grid of 4 CTAs of 512
 * threads per SM runs 8 independent FMA chains per thread, as scalar fma.rn.f32 (paired = 0) or
 * as paired fma.rn.f32x2 instructions (paired = 1, two FMAs each); *fma_per_s receives the best
 * of three timed launches (CUDA events), in FMAs per second.  Clocks are left as they are. */
int aecct_selftest_fma_rate(int32_t paired, double *fma_per_s);

#ifdef __cplusplus
}
#endif

#endif /* AECCT_H */
