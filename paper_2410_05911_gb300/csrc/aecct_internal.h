// aecct_internal.h -- parameters shared by the host side (api.cu) and the decoder kernel
// (decoder_kernel.cuh) of libaecct.  Not part of the public ABI.
#pragma once
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <cstdint>

namespace aecct {

constexpr int kRows = 128;          // token rows per CTA: one M = 128 tensor-core tile
constexpr int kHeads = 8;           // this build: 8 attention heads
constexpr int kEpiWarps = 16;       // 4 TMEM lane quadrants x 4 column slices
constexpr int kEpiThreads = kEpiWarps * 32;
constexpr int kThreads = kEpiThreads;  // warp 0 also streams weights and issues the MMAs
constexpr int kMaxCluster = 8;
constexpr int kOutBitsBytes = 4096;      // decoded bits of the codewords one CTA finishes
constexpr int kMaxTasks = 16;            // attention tasks per warp (task mode)
constexpr int kQSlots = 8;               // d = 128 tasks run off their quadrant (2 KB Q/A slots in W2)
constexpr int kMaxGroups = 32;           // 32-row query groups per CTA (task mode)
constexpr int kTaskCache = 64;           // attention scores per task kept in TMEM (task mode)
constexpr int kRowCache = 64;            // attention scores per (row, head) kept in TMEM (row mode)

// One weight chunk of a block: rows [n0, n0 + nrows) and K columns [k0, k0 + kcols) of the
// block's GEMM `gemm` (0 = QKV, 1 = O, 2 = FFN1, 3 = FFN2), stored as a K-major bf16 tile
// of 8 x 16-byte core matrices at byte offset `off` of the block's weight stream.
struct ChunkDesc {
  uint32_t off;
  uint32_t bytes;
  int gemm, n0, nrows, k0, kcols;
};

// The fixed order in which a block's weights stream through shared memory, for model width D.
// GEMM g has N_g output rows and K_g inputs: QKV (3D, D), O (D, D), FFN1 (4D, D), FFN2 (D, 4D).
// D = 32 and 64: one chunk per GEMM (N <= 256 is a single tcgen05.mma shape), two stages of the
// largest GEMM.  D = 128: 128 x 64 chunks, three 16 KB stages.  A block has kCPL chunks; kCPL is
// a multiple of 2 kStages, so chunk p of any block uses stage p % kStages and completes phase
// parity (p / kStages) & 1 of that stage's barriers, whatever block it belongs to.
template <int D>
struct WeightSchedule {
  static constexpr int kStages = (D == 128) ? 3 : 2;
  static constexpr uint32_t kStageBytes = (D == 32) ? 8192u : (D == 64) ? 32768u : 16384u;
  __host__ __device__ static constexpr int gemm_n(int g) { return g == 0 ? 3 * D : (g == 2 ? 4 * D : D); }
  __host__ __device__ static constexpr int gemm_k(int g) { return g == 3 ? 4 * D : D; }
  __host__ __device__ static constexpr int tile_n(int g) { return D == 128 ? 128 : gemm_n(g); }
  __host__ __device__ static constexpr int tile_k(int g) { return D == 128 ? 64 : gemm_k(g); }
  __host__ __device__ static constexpr int count(int g) {
    return ((gemm_n(g) + tile_n(g) - 1) / tile_n(g)) * (gemm_k(g) / tile_k(g));
  }
  __host__ __device__ static constexpr int first(int g) {
    int f = 0;
    for (int h = 0; h < g; ++h) f += count(h);
    return f;
  }
  static constexpr int kCPL = first(4);  // chunks per block
  // N tile and K tile of chunk j of GEMM g.  N tiles go in pairs, a pair's two chunks of one K
  // range adjacent (two 128-row tiles form one 256-row operand for an N = 256 MMA); an odd last N
  // tile follows with its K tiles in order.
  __host__ __device__ static constexpr int tile_of(int g, int j, bool want_n) {
    const int nt = (gemm_n(g) + tile_n(g) - 1) / tile_n(g), kt = gemm_k(g) / tile_k(g);
    const int paired = (nt / 2) * 2 * kt;
    int n = 0, k = 0;
    if (j < paired) {
      n = 2 * (j / (2 * kt)) + (j % 2);
      k = (j % (2 * kt)) / 2;
    } else {
      n = nt - 1;
      k = j - paired;
    }
    return want_n ? n : k;
  }
  __host__ __device__ static constexpr ChunkDesc chunk(int p) {
    int g = 0;
    while (g < 3 && p >= first(g + 1)) ++g;
    const int j = p - first(g);
    const int n0 = tile_of(g, j, true) * tile_n(g), k0 = tile_of(g, j, false) * tile_k(g);
    const int nrows = (gemm_n(g) - n0) < tile_n(g) ? (gemm_n(g) - n0) : tile_n(g);
    uint32_t off = 0;
    for (int q = 0; q < p; ++q) off += chunk_bytes(q);
    return ChunkDesc{off, static_cast<uint32_t>(nrows * tile_k(g) * 2), g, n0, nrows, k0, tile_k(g)};
  }
  __host__ __device__ static constexpr uint32_t chunk_bytes(int p) {
    int g = 0;
    while (g < 3 && p >= first(g + 1)) ++g;
    const int j = p - first(g);
    const int n0 = tile_of(g, j, true) * tile_n(g);
    const int nrows = (gemm_n(g) - n0) < tile_n(g) ? (gemm_n(g) - n0) : tile_n(g);
    return static_cast<uint32_t>(nrows * tile_k(g) * 2);
  }
  static constexpr uint32_t kLayerBytes = chunk(kCPL - 1).off + chunk_bytes(kCPL - 1);
};
// d = 128: the hidden unit whose FFN1 accumulator sits in TMEM column c (the weight row that the
// weight stream places at FFN1 output column c).  Column slice s of a row owns hidden units
// [128 s, 128 s + 128): units 128 s + [0, 64) in columns [64 s, 64 s + 64), done with FFN1's first
// N-tile pair, and units 128 s + [64, 128) in columns [256 + 64 s, 256 + 64 s + 64).  The FFN2
// operand codes of unit h, two to a 32-bit column, then go to column h / 2, which lies in the
// slice's own first range and was read before it is written; FFN2's accumulators take [256, 384).
// Other widths keep the identity.
__host__ __device__ constexpr int ffn1_unit_of_column(int D, int c) {
  return D == 128 ? 128 * ((c % 256) / 64) + 64 * (c / 256) + (c % 64) : c;
}

// the tcgen05.mma shape rules (M = 128: 16 <= N <= 256, N % 16 == 0) and the stage sizes
template <int D>
__host__ __device__ constexpr bool schedule_ok() {
  using W = WeightSchedule<D>;
  if (W::kCPL % (2 * W::kStages) != 0) return false;
  for (int p = 0; p < W::kCPL; ++p) {
    const ChunkDesc c = W::chunk(p);
    if (c.nrows < 16 || c.nrows > 256 || c.nrows % 16 != 0 || c.kcols % 16 != 0) return false;
    if (c.bytes > W::kStageBytes || c.off % 16 != 0) return false;
  }
  return true;
}
static_assert(schedule_ok<32>() && schedule_ok<64>() && schedule_ok<128>(), "weight schedule");

// Per-block parameter vector layout (floats), D = model width.
struct LayerParamLayout {
  __host__ __device__ static constexpr int bqkv(int) { return 0; }        // b_q | b_k | b_v  (3D)
  __host__ __device__ static constexpr int bo(int D) { return 3 * D; }     // b_o (D)
  __host__ __device__ static constexpr int b1(int D) { return 4 * D; }     // b_1 (4D)
  __host__ __device__ static constexpr int b2(int D) { return 8 * D; }     // b_2 (D)
  __host__ __device__ static constexpr int ln1g(int D) { return 9 * D; }
  __host__ __device__ static constexpr int ln1b(int D) { return 10 * D; }
  __host__ __device__ static constexpr int ln2g(int D) { return 11 * D; }
  __host__ __device__ static constexpr int ln2b(int D) { return 12 * D; }
  __host__ __device__ static constexpr int sw(int D) { return 13 * D; }    // 6 scales gamma*delta (+2 pad)
  __host__ __device__ static constexpr int stride(int D) { return 13 * D + 8; }
};

struct DecodeParams {
  // problem shape
  int n, k, T, m, n_layers, h_first, d_spe;
  int Tp;          // token rows per codeword: T, or more when the rows of each node type start on a
                   // 32-row boundary (d = 128 warp tasks); a padding row holds no token (perm 0xFFFF)
  int C;           // CTAs per cluster (they share one group of codewords)
  int G;           // codewords per group
  int n_clusters;  // clusters launched
  int64_t B, n_groups;
  // inputs / outputs (device)
  const float *y;
  uint8_t *bits;
  uint8_t *syn;
  float *logits;
  // model (device)
  const uint8_t *wstream;  // bf16 weight chunks in WeightSchedule<D> order, block after block
  uint32_t layer_bytes;    // WeightSchedule<D>::kLayerBytes
  const float *lparams;  // [n_layers][LayerParamLayout::stride(D)]
  const float *emb;      // [T][D - d_spe]
  const float *spe;      // [T][d_spe]
  const float *w_d1;     // [D]
  float b_d1;
  const float *w_out;    // [T][n]
  const float *b_out;    // [n]
  const uint32_t *hbits;  // [m][hwords] row i of H as a bitmask over the variables (bit j%32 of word j/32)
  int hwords;             // ceil(n / 32)
  const uint16_t *perm;         // [Tp] row offset within a codeword -> token (0xFFFF: padding row)
  const uint16_t *pos;          // [T] token -> row offset within its codeword
  // HPSA neighbour lists, 0 = first ring, 1 = second ring.  mask_info[mk][t] = (start << 11) | count:
  // the count row offsets of token t's neighbours (ascending token order) begin at mask_list[mk][start]
  // and continue 8 per 16-byte entry (a list is padded to whole entries).
  const uint32_t *mask_info[2];
  const uint4 *mask_list[2];
  // Task-mode attention plan (one CTA per group of codewords, d <= 64).  A task is one head for
  // a query group: up to 32 consecutive rows of one codeword, one per lane.  It walks the union of
  // its lanes' key sets (ascending token order) with per-lane membership bits.
  // The plan is one blob that every CTA copies into shared memory (after the SmemLayout regions)
  // at the start of the kernel; the offsets are byte offsets into it, 16-byte aligned:
  //   task  [16 warps][kMaxTasks] uint16: group * 8 + head; 0xFFFF ends the list
  //   grp   [groups] uint4: {first row, lanes, first row of the codeword, 0}
  //   uinfo [groups][2 rings] uint32: (start << 8) | count of the union list
  //   ulist union lists: 16 row offsets (one byte each) per 16-byte entry
  //   mask  [groups][2][32 lanes] uint4: 128 membership bits over the union list
  //   qslot (d = 128) uint8 [4] group of each TMEM lane quadrant (0xFF: none), then
  //         [groups][8 heads] the Q/A slot of the task (group, head): 0xFF when it runs on a warp of
  //         its group's quadrant (Q and A in TMEM), else a 2 KB slot of weight stage W2
  const uint4 *plan_blob;
  uint32_t plan_bytes;  // a multiple of 16; 0 without warp tasks
  uint32_t off_task, off_grp, off_uinfo, off_ulist, off_mask, off_qslot;

  float ln_eps, alpha_floor, att_scale;
  int alpha_mode;  // 0 = absmax alpha per token row, 1 = per quantised matrix of a word (C == 1)
  // integer-core capture (device, optional)
  int64_t cap_B;
  int8_t *cap_q;
  int32_t *cap_acc;
  float *cap_alpha;
  uint8_t *cap_syn;
  // staged attention (d = 128): K and V of every row, per cluster, in global memory (L2), read back
  // head by head with bulk copies: [cluster][8 heads][K, V][C * 128 rows][16 floats], 16-byte
  // piece f of row rho at f ^ ((rho >> 1) & 3)
  float *kv_scratch;
  // control
  int *err;  // device word, bit 0 = a bounded wait timed out
  long long wait_limit;
};

// Byte offset of element (r, c) in a K-major no-swizzle operand tile whose rows hold kdim
// elements of 2 bytes: core matrix (r/8, c/8) is 128 contiguous bytes, core matrices along
// K are adjacent (lbo = 128), 8-row groups are kdim/8 * 128 bytes apart (sbo).
__host__ __device__ constexpr inline uint32_t core_off(uint32_t r, uint32_t c, uint32_t kdim) {
  return (r >> 3) * (kdim >> 3) * 128u + (c >> 3) * 128u + (r & 7u) * 16u + (c & 7u) * 2u;
}

// Shared-memory map.  Region U holds, per block, first the attention operands and then the FFN2
// operand.  Row mode, and task mode at d = 128: per token row 8 heads x (K | V) x d_h fp32 (Q and
// the attention output stay in TMEM).  Task mode at d <= 64: 8 heads x (Q | K | V) x d_h fp32;
// the attention output of a (row, head) then replaces its Q.
template <int D, bool TASKS = false>
struct SmemLayout {
  static constexpr bool kQInSmem = TASKS && D != 128;
  static constexpr uint32_t kSlot = (kQInSmem ? 12u : 8u) * (D / 8u);  // bytes of one head of one row
  static constexpr uint32_t kKvStride = 8u * kSlot + 16u;            // token row, + 16 B pad
  static constexpr uint32_t kKvBytes = kRows * kKvStride;
  static constexpr uint32_t kUqBytes = kRows * 4u * D * 2u;  // FFN2 operand: 128 x 4D bf16
  __host__ __device__ static constexpr uint32_t align1k(uint32_t v) { return (v + 1023u) & ~1023u; }
  static constexpr uint32_t kRegionU = align1k(kKvBytes > kUqBytes ? kKvBytes : kUqBytes);
  static constexpr uint32_t kAopBytes = kRows * D * 2u;  // QKV / O / FFN1 operand: 128 x D bf16
  static constexpr int kStages = WeightSchedule<D>::kStages;
  static constexpr uint32_t kStageBytes = WeightSchedule<D>::kStageBytes;
  static constexpr uint32_t kOffU = 0;
  static constexpr uint32_t kOffAop = kRegionU;
  static constexpr uint32_t kOffW = align1k(kOffAop + kAopBytes);
  static constexpr uint32_t kOffRed = kOffW + kStages * kStageBytes;  // 2 x 4 x 128 floats
  static constexpr uint32_t kOffZ = kOffRed + 4096;                   // 128 floats
  static constexpr uint32_t kOffObits = kOffZ + 512;                  // decoded bits
  static constexpr uint32_t kOffBitWords = kOffObits + kOutBitsBytes;  // 128 words: bitmasks of a group's words
  static constexpr uint32_t kOffBar = kOffBitWords + 512;              // mbarriers
  static constexpr uint32_t kOffMisc = kOffBar + 256;  // tmem base, abort flag, peer bases, copy count
  static constexpr uint32_t kTotal = kOffMisc + 256;
  // QKV / FFN1 accumulators in [0, 4D) (x parked in [3D, 4D) during attention).  Attention
  // scores are cached in TMEM between the two softmax passes: task mode from kTaskCacheCol
  // (4 warps per lane quadrant x kTaskCache columns: [256, 512) for d <= 64, the dead K and V
  // accumulator columns [128, 384) for d = 128); row mode kRowCache columns per column slice
  // from kRowCacheCol, each thread in its own row's lane (d = 128: [128, 384); d <= 64:
  // [256, 512)).
  static constexpr uint32_t kTmemCols = 512u;
  static constexpr uint32_t kTaskCacheCol = (D == 128) ? 128u : 256u;
  static constexpr uint32_t kRowCacheCol = (D == 128) ? 128u : 256u;
};

// decoder_kernel.cuh.  ATT: 0 = per-row neighbour lists, 1 = warp tasks, 2 = per-row lists over
// per-head staged rows (d = 128); ACT: 0 = ReLU, 1 = GELU; LIN: 0 = AAP linears, 1 = full-precision
// (bf16) linears.  Instantiated in decoder_kernel.cu (0, 0), decoder_kernel_gelu.cu (1, 0),
// decoder_kernel_fp.cu (0, 1) and decoder_kernel_fp_gelu.cu (1, 1).
template <int D, int ATT, int ACT, int LIN>
cudaError_t launch_decode(const DecodeParams &p, cudaStream_t stream);
template <int D, int ATT, int ACT, int LIN>
cudaError_t prepare_decode_kernel(int cluster_ctas, uint32_t plan_bytes, int *max_active_clusters);
constexpr uint32_t kMaxDynSmem = 232448;  // the largest dynamic shared memory a CTA may opt into (227 KB)
constexpr int kStagedMaxRows = 640;  // staged attention: rows of a group (64 bytes of K and of V each, 40 KB + 40 KB)
constexpr int kStagedMaxKeys = 256;  // staged attention: keys per row (TMEM columns [128, 384))

// aap.cu: the AAP weight quantiser (eq. Ternary) and the GPU expansion of 2-bit weights
constexpr int kTernarizeMaxTensors = 64;  // tensors per launch (the launcher splits larger calls)
cudaError_t launch_aap_ternarize(const float *w, int n, const int64_t *len, const float *delta, float eps,
                                 uint8_t *packed, float *scale, float *wq, cudaStream_t stream);
cudaError_t launch_unpack_weights(const uint8_t *packed, int n_layers, int D, const ChunkDesc *chunks, int n_chunks,
                                  uint32_t layer_bytes, uint8_t *wstream, cudaStream_t stream);

// spe.cu: the spectral positional encoding (Sec. 4.3) on the GPU
constexpr int kSpeMaxHeads = 8;
constexpr int kSpeMaxTokens = 1024;
cudaError_t run_spe_table(const uint8_t *H, int n, int m, int d_spe, int heads, const double *w_pe, const double *wq,
                          const double *wk, const double *wv, const double *wo, double cluster_tol, double vanish_tol,
                          float *spe_host, double *lam_host, double *U_host, double *spe64_host, int *sweeps,
                          int *status_host);

// api.cu diagnostics kernels live in selftest.cu
cudaError_t run_selftest_mma(const int8_t *a_host, const int8_t *b_host, int K, int N, float *out_host);
cudaError_t run_selftest_timeout(long long limit_cycles, int *status_host);
cudaError_t run_selftest_fma_rate(bool paired, double *fma_per_s);

}  // namespace aecct
