// api.cu -- host side of libaecct's C ABI (include/aecct.h).
//
// aecct_create validates the model description, builds the HPSA neighbour lists from H
// (Sec. 4.2), unpacks the 2-bit ternary weights into bf16 tensor-core tiles, picks how many
// CTAs share a group of codewords, and copies everything to the device once.  aecct_decode
// launches the fused decoder kernel (decoder_kernel.cuh) on the caller's stream.
#include <cuda_runtime.h>

#include <cmath>
#include <cstdlib>
#include <algorithm>
#include <cstring>
#include <string>
#include <vector>

#include "../../include/aecct.h"
#include "aecct_internal.h"

using namespace aecct;

namespace {

thread_local std::string g_last_error;

int cuda_fail(cudaError_t e, const char *what) {
  g_last_error = std::string(what) + ": " + cudaGetErrorString(e);
  return AECCT_ERR_CUDA;
}

}  // namespace

struct aecct_handle {
  int n = 0, k = 0, T = 0, m = 0, d = 0, n_layers = 0, h_first = 0, d_spe = 0;
  int Tp = 0;  // token rows per codeword (T, or T plus padding rows)
  int C = 1, G = 1, max_clusters = 0;
  int att = 0;  // kernel attention path: 0 per-row lists, 1 warp tasks, 2 per-row lists over staged rows
  int alpha_mode = 0;  // 1 = one alpha per quantised matrix of a word
  int activation = 0;   // 0 = ReLU, 1 = GELU
  int linear_mode = 0;  // 0 = AAP ternary linears, 1 = full-precision (bf16) linears
  float ln_eps = 0, alpha_floor = 0, att_scale = 0, b_d1 = 0;
  long long wait_limit = 0;
  int device = 0;
  std::vector<void *> allocs;
  uint8_t *wstream = nullptr;
  uint32_t layer_bytes = 0;
  int n_chunks = 0;
  ChunkDesc chunks[32] = {};  // WeightSchedule<d> order
  float *lparams = nullptr, *emb = nullptr, *spe = nullptr, *w_d1 = nullptr, *w_out = nullptr, *b_out = nullptr;
  uint32_t *hbits = nullptr, *mask_info[2] = {nullptr, nullptr};
  int hwords = 0;
  uint16_t *mask_list[2] = {nullptr, nullptr};
  uint16_t *perm = nullptr, *pos = nullptr;
  float *kv_scratch = nullptr;  // staged attention: K and V rows per cluster
  uint8_t *plan_blob = nullptr;  // the attention plan (task mode), copied into shared memory by the kernel
  uint32_t plan_bytes = 0, off_task = 0, off_grp = 0, off_uinfo = 0, off_ulist = 0, off_mask = 0, off_qslot = 0;
  int *d_err = nullptr;
  int *h_err = nullptr;  // pinned
  cudaEvent_t ev = nullptr;
  bool ev_pending = false;
  int pending_status = AECCT_OK;
  // capture
  int64_t cap_B = 0;
  int8_t *cap_q = nullptr;
  int32_t *cap_acc = nullptr;
  float *cap_alpha = nullptr;
  uint8_t *cap_syn = nullptr;
  // host-buffer staging
  int64_t stage_B = 0;
  float *st_y = nullptr, *st_logits = nullptr;
  uint8_t *st_bits = nullptr, *st_syn = nullptr;
};

namespace {

template <typename T>
int dev_upload(aecct_handle *h, T **dst, const T *src, size_t count) {
  void *p = nullptr;
  const size_t bytes = sizeof(T) * (count ? count : 1);
  cudaError_t e = cudaMalloc(&p, bytes);
  if (e != cudaSuccess) return e == cudaErrorMemoryAllocation ? AECCT_ERR_OUT_OF_MEMORY : cuda_fail(e, "cudaMalloc");
  h->allocs.push_back(p);
  if (count && src) {
    e = cudaMemcpy(p, src, sizeof(T) * count, cudaMemcpyHostToDevice);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpy");
  }
  *dst = static_cast<T *>(p);
  return AECCT_OK;
}

void free_handle(aecct_handle *h) {
  if (!h) return;
  for (void *p : h->allocs) cudaFree(p);
  cudaFree(h->st_y);
  cudaFree(h->st_logits);
  cudaFree(h->st_bits);
  cudaFree(h->st_syn);
  if (h->h_err) cudaFreeHost(h->h_err);
  if (h->ev) cudaEventDestroy(h->ev);
  delete h;
}

// bf16 encoding of a finite fp32 value, rounded to nearest even (the low 16 bits decide; a tie
// goes to the even upper half)
uint16_t bf16_rne_bits(float f) {
  uint32_t u;
  std::memcpy(&u, &f, 4);
  u += 0x7FFFu + ((u >> 16) & 1u);
  return static_cast<uint16_t>(u >> 16);
}

uint16_t f2bf_bits(float f) {
  // exact for the integers -1, 0, 1
  uint32_t u;
  std::memcpy(&u, &f, 4);
  return static_cast<uint16_t>(u >> 16);
}

int validate(const aecct_model_desc *d) {
  if (!d) return AECCT_ERR_INVALID_ARG;
  if (d->n <= 0 || d->k <= 0 || d->k >= d->n) return AECCT_ERR_INVALID_ARG;
  if (d->d <= 0 || d->heads <= 0 || d->d % d->heads != 0) return AECCT_ERR_INVALID_ARG;
  if (d->n_layers < 1 || d->n_layers > 4096) return AECCT_ERR_INVALID_ARG;
  if (d->h_first < 0 || d->h_first > d->heads) return AECCT_ERR_INVALID_ARG;
  if (d->d_spe < 0 || d->d_spe >= d->d) return AECCT_ERR_INVALID_ARG;
  if (d->ffn_mult <= 0) return AECCT_ERR_INVALID_ARG;
  if (d->activation < 0 || d->activation > 1) return AECCT_ERR_INVALID_ARG;
  if (d->cluster_ctas < 0 || d->cluster_ctas > 64) return AECCT_ERR_INVALID_ARG;
  if (d->attention_mode < 0 || d->attention_mode > 3) return AECCT_ERR_INVALID_ARG;
  if (d->mask_mode < 0 || d->mask_mode > 1) return AECCT_ERR_INVALID_ARG;
  if (d->alpha_mode < 0 || d->alpha_mode > 1) return AECCT_ERR_INVALID_ARG;
  if (d->linear_mode < 0 || d->linear_mode > 1) return AECCT_ERR_INVALID_ARG;
  const bool aap = d->linear_mode == 0;
  if (!aap && d->alpha_mode != 0) return AECCT_ERR_INVALID_ARG;  // alpha belongs to eq. Quant
  if (aap && (!d->w_packed || !d->w_scale)) return AECCT_ERR_INVALID_ARG;
  if (!aap && !d->w_full) return AECCT_ERR_INVALID_ARG;
  if (!d->H || !d->emb || !d->bias || !d->ln_gamma || !d->ln_beta || !d->w_d1 || !d->w_out || !d->b_out)
    return AECCT_ERR_INVALID_ARG;
  if (d->d_spe > 0 && !d->spe) return AECCT_ERR_INVALID_ARG;
  if (!(d->ln_eps >= 0.0f) || !std::isfinite(d->ln_eps)) return AECCT_ERR_INVALID_ARG;
  if (!(d->alpha_floor > 0.0f) || !std::isfinite(d->alpha_floor)) return AECCT_ERR_INVALID_ARG;
  if (d->wait_limit_cycles < 0) return AECCT_ERR_INVALID_ARG;
  const int n = d->n, m = d->n - d->k;
  for (int i = 0; i < m; ++i) {
    int row = 0;
    for (int j = 0; j < n; ++j) {
      const uint8_t v = d->H[(size_t)i * n + j];
      if (v > 1) return AECCT_ERR_INVALID_ARG;
      row += v;
    }
    if (row == 0) return AECCT_ERR_INVALID_ARG;
  }
  for (int j = 0; j < n; ++j) {
    int col = 0;
    for (int i = 0; i < m; ++i) col += d->H[(size_t)i * n + j];
    if (col == 0) return AECCT_ERR_INVALID_ARG;
  }
  // shape limits of this build
  if (d->heads != kHeads) return AECCT_ERR_UNSUPPORTED;
  if (d->d != 32 && d->d != 64 && d->d != 128) return AECCT_ERR_UNSUPPORTED;
  if (d->ffn_mult != 4) return AECCT_ERR_UNSUPPORTED;
  const int T = 2 * n - d->k;
  if (T > kMaxCluster * kRows || T > 65535) return AECCT_ERR_UNSUPPORTED;
  // packed weights: no code 10; full-precision weights: finite
  if (!aap) {
    const size_t nw = (size_t)d->n_layers * 12u * d->d * d->d;
    for (size_t i = 0; i < nw; ++i)
      if (!std::isfinite(d->w_full[i])) return AECCT_ERR_INVALID_ARG;
    return AECCT_OK;
  }
  const size_t nbytes = (size_t)d->n_layers * 12u * d->d * d->d / 4u;
  for (size_t i = 0; i < nbytes; ++i) {
    const uint8_t b = d->w_packed[i];
    for (int s = 0; s < 4; ++s)
      if (((b >> (2 * s)) & 3u) == 2u) return AECCT_ERR_INVALID_ARG;
  }
  return AECCT_OK;
}

// 2-bit code -> ternary value
inline int8_t tern(uint8_t code) { return code == 1 ? 1 : (code == 3 ? -1 : 0); }

struct Gemm {
  int N, K;
};

// the chunks of one block in the order the kernel streams them (WeightSchedule<D>)
template <int D>
int schedule_chunks_t(ChunkDesc *out) {
  using W = WeightSchedule<D>;
  static_assert(W::kCPL <= 32, "chunk table");
  for (int c = 0; c < W::kCPL; ++c) out[c] = W::chunk(c);
  return W::kCPL;
}
int schedule_chunks(int D, ChunkDesc *out) {
  return D == 32 ? schedule_chunks_t<32>(out) : D == 64 ? schedule_chunks_t<64>(out) : schedule_chunks_t<128>(out);
}

// ---- warp-task attention plan: which warp runs which task
// A task (one head for one query group) costs the length of its union key list + 4 (its fixed
// part).  Warps w with the same w % 4 issue from one scheduler and share its issue slots.  Measured
// on the GPU: a warp alone issues at about 0.36 of a scheduler's rate (its own dependency chains
// limit it) and about three warps saturate a scheduler, so four warps with unequal loads leave a
// tail where one warp runs alone (Polar(64,32): its tasks on three warps per scheduler decode 2.2%
// faster than on four; BCH(63,36)'s on two warps per lane quadrant instead of four make the
// attention 1.38x slower).  A scheduler's time is modelled in phases: while k of its warps have
// work left, each advances at min(1, k s) / k.  The plan minimises the largest modelled time.
constexpr double kWarpIssueShare = 0.36;

double scheduler_time(std::vector<long> loads) {
  loads.erase(std::remove(loads.begin(), loads.end(), 0L), loads.end());
  std::sort(loads.begin(), loads.end());
  double t = 0.0;
  long done = 0;
  const int n = static_cast<int>(loads.size());
  for (int i = 0; i < n; ++i) {
    const int k = n - i;  // warps with work left
    const double per_warp = std::min(1.0, k * kWarpIssueShare) / k;
    t += static_cast<double>(loads[i] - done) / per_warp;
    done = loads[i];
  }
  return t;
}

// The tasks of one scheduler (costs in descending order) onto its four warps, minimising
// scheduler_time: every assignment for up to 9 tasks (a task opens at most the first empty warp,
// which skips permutations of equivalent warps), else the best of longest-first onto 1..4 warps.
// out[i] is the warp slot (0..3) of task i; false if no assignment keeps each warp within `cap`.
bool assign_scheduler(const std::vector<int> &cost, int cap, std::vector<int> &out, double *time = nullptr) {
  const int m = static_cast<int>(cost.size());
  out.assign(m, 0);
  if (time) *time = 0.0;
  if (m == 0) return true;
  double best = 1e300;
  std::vector<int> cur(m, 0);
  if (m <= 9) {
    long load[4] = {0, 0, 0, 0};
    int cnt[4] = {0, 0, 0, 0};
    auto rec = [&](auto &&self, int i, int used) -> void {
      if (i == m) {
        const double t = scheduler_time({load[0], load[1], load[2], load[3]});
        if (t < best) best = t, out = cur;
        return;
      }
      for (int w = 0; w < std::min(used + 1, 4); ++w) {
        if (cnt[w] >= cap) continue;
        load[w] += cost[i], ++cnt[w], cur[i] = w;
        self(self, i + 1, std::max(used, w + 1));
        load[w] -= cost[i], --cnt[w];
      }
    };
    rec(rec, 0, 0);
  } else {
    for (int k = 1; k <= 4; ++k) {
      std::vector<long> load(k, 0);
      std::vector<int> cnt(k, 0);
      bool ok = true;
      for (int i = 0; i < m && ok; ++i) {
        int b = -1;
        for (int w = 0; w < k; ++w)
          if (cnt[w] < cap && (b < 0 || load[w] < load[b])) b = w;
        if (b < 0) ok = false;
        else load[b] += cost[i], ++cnt[b], cur[i] = b;
      }
      if (!ok) continue;
      const double t = scheduler_time(load);
      if (t < best) best = t, out = cur;
    }
  }
  if (time) *time = best;
  return best < 1e300;
}

// the compiled kernel for (d, attention path ATT, activation ACT, linear mode LIN)
template <int ACT, int LIN>
cudaError_t prepare_any(int D, int att, int C, uint32_t pb, int *max_clusters) {
  if (att == 1)
    return D == 32   ? prepare_decode_kernel<32, 1, ACT, LIN>(C, pb, max_clusters)
           : D == 64 ? prepare_decode_kernel<64, 1, ACT, LIN>(C, pb, max_clusters)
                     : prepare_decode_kernel<128, 1, ACT, LIN>(C, pb, max_clusters);
  if (att == 2) return prepare_decode_kernel<128, 2, ACT, LIN>(C, pb, max_clusters);  // d = 128 only
  if (D == 32) return prepare_decode_kernel<32, 0, ACT, LIN>(C, pb, max_clusters);
  if (D == 64) return prepare_decode_kernel<64, 0, ACT, LIN>(C, pb, max_clusters);
  return prepare_decode_kernel<128, 0, ACT, LIN>(C, pb, max_clusters);
}
template <int ACT, int LIN>
cudaError_t launch_any(int D, int att, const DecodeParams &p, cudaStream_t stream) {
  if (att == 1)
    return D == 32   ? launch_decode<32, 1, ACT, LIN>(p, stream)
           : D == 64 ? launch_decode<64, 1, ACT, LIN>(p, stream)
                     : launch_decode<128, 1, ACT, LIN>(p, stream);
  if (att == 2) return launch_decode<128, 2, ACT, LIN>(p, stream);
  if (D == 32) return launch_decode<32, 0, ACT, LIN>(p, stream);
  if (D == 64) return launch_decode<64, 0, ACT, LIN>(p, stream);
  return launch_decode<128, 0, ACT, LIN>(p, stream);
}
cudaError_t prepare_variant(int act, int lin, int D, int att, int C, uint32_t pb, int *max_clusters) {
  if (lin == 0)
    return act == 0 ? prepare_any<0, 0>(D, att, C, pb, max_clusters) : prepare_any<1, 0>(D, att, C, pb, max_clusters);
  return act == 0 ? prepare_any<0, 1>(D, att, C, pb, max_clusters) : prepare_any<1, 1>(D, att, C, pb, max_clusters);
}
cudaError_t launch_variant(int act, int lin, int D, int att, const DecodeParams &p, cudaStream_t stream) {
  if (lin == 0) return act == 0 ? launch_any<0, 0>(D, att, p, stream) : launch_any<1, 0>(D, att, p, stream);
  return act == 0 ? launch_any<0, 1>(D, att, p, stream) : launch_any<1, 1>(D, att, p, stream);
}

}  // namespace

extern "C" {

const char *aecct_status_string(int status) {
  switch (status) {
    case AECCT_OK: return "ok";
    case AECCT_ERR_INVALID_ARG: return "invalid argument";
    case AECCT_ERR_UNSUPPORTED: return "unsupported model shape for this build";
    case AECCT_ERR_OUT_OF_MEMORY: return "out of device memory";
    case AECCT_ERR_CUDA: return "CUDA error";
    case AECCT_ERR_TIMEOUT: return "device-side wait timed out";
    case AECCT_ERR_NO_DEVICE: return "no sm_103 device";
    default: return "unknown status";
  }
}

const char *aecct_last_error(void) { return g_last_error.c_str(); }

int aecct_create(const aecct_model_desc *desc, aecct_handle **out) {
  if (!out) return AECCT_ERR_INVALID_ARG;
  *out = nullptr;
  int rc = validate(desc);
  if (rc) return rc;
  const aecct_model_desc &d = *desc;
  const int n = d.n, k = d.k, m = n - k, T = 2 * n - k, D = d.d, F = 4 * D;

  // ---- HPSA neighbour lists (Sec. 4.2): token t < n is variable t, token n + i is check i.
  // First ring: Tanner-graph neighbours.  Second ring: same-type nodes at distance two, and the
  // node itself.  Lists are in ascending token order (the order the softmax sums run in).
  std::vector<std::vector<uint16_t>> nb[2];
  nb[0].resize(T);
  nb[1].resize(T);
  {
    std::vector<uint8_t> row(T);
    for (int t = 0; t < T; ++t) {
      std::fill(row.begin(), row.end(), 0);
      if (t < n) {
        for (int i = 0; i < m; ++i)
          if (d.H[(size_t)i * n + t]) row[n + i] = 1;
      } else {
        for (int j = 0; j < n; ++j)
          if (d.H[(size_t)(t - n) * n + j]) row[j] = 1;
      }
      for (int u = 0; u < T; ++u)
        if (row[u]) nb[0][t].push_back(static_cast<uint16_t>(u));
      std::fill(row.begin(), row.end(), 0);
      if (t < n) {
        for (int i = 0; i < m; ++i)
          if (d.H[(size_t)i * n + t])
            for (int j = 0; j < n; ++j)
              if (d.H[(size_t)i * n + j]) row[j] = 1;
      } else {
        const int i0 = t - n;
        for (int j = 0; j < n; ++j)
          if (d.H[(size_t)i0 * n + j])
            for (int i = 0; i < m; ++i)
              if (d.H[(size_t)i * n + j]) row[n + i] = 1;
      }
      for (int u = 0; u < T; ++u)
        if (row[u]) nb[1][t].push_back(static_cast<uint16_t>(u));
    }
  }
  if (d.mask_mode == 1) {
    // ECCT code-aware mask (Sec. 3) for every head: the union of the two rings, ascending
    for (int t = 0; t < T; ++t) {
      std::vector<uint16_t> u;
      std::merge(nb[0][t].begin(), nb[0][t].end(), nb[1][t].begin(), nb[1][t].end(), std::back_inserter(u));
      u.erase(std::unique(u.begin(), u.end()), u.end());
      nb[0][t] = u;
      nb[1][t] = u;
    }
  }

  // Attention mode.  Task mode keeps every codeword inside one CTA (no cluster).  d <= 64: Q, K, V
  // and A in shared memory, T <= 128, at most kMaxGroups 32-row query groups.  d = 128: Q and A in
  // TMEM, one codeword per CTA whose variables start at row 0 and whose checks start on the next
  // 32-row boundary, so that every query group is one TMEM lane quadrant (Tp = that padded row
  // count <= 128), one alpha per row.  By default d = 128 takes task mode only when the query
  // groups' shared key lists are dense enough that walking their unions beats walking each
  // row's own list.
  const int g1 = kRows / T;
  const int npad = ((n + 31) / 32) * 32, Tp128 = npad + m;
  const bool one_cta = d.cluster_ctas == 0 || d.cluster_ctas == 1;
  const bool task_ok =
      D <= 64 ? (T <= kRows && g1 >= 1 && g1 * ((T + 31) / 32) <= kMaxGroups && g1 * n <= kOutBitsBytes && one_cta)
              : (Tp128 <= kRows && d.alpha_mode == 0 && n <= kOutBitsBytes && one_cta);
  bool tasks = false;
  if (d.attention_mode == 2) {
    if (!task_ok) return AECCT_ERR_UNSUPPORTED;
    tasks = true;
  } else if (d.attention_mode == 0) {
    tasks = task_ok;
    if (tasks && D == 128) {
      // share of the lane-key iterations of the task walks that fall on a lane's own keys
      double useful = 0.0, walked = 0.0;
      const int hr[2] = {d.h_first, d.heads - d.h_first};
      for (int r = 0; r < 2; ++r) {
        for (int t = 0; t < T; ++t) useful += hr[r] * static_cast<double>(nb[r][t].size());
        for (int type = 0; type < 2; ++type) {
          const int t0 = type == 0 ? 0 : n, t1 = type == 0 ? n : T;
          for (int g0 = t0; g0 < t1; g0 += 32) {
            std::vector<uint8_t> in(T, 0);
            int u = 0;
            for (int t = g0; t < std::min(g0 + 32, t1); ++t)
              for (uint16_t v : nb[r][t]) u += in[v] ? 0 : (in[v] = 1);
            walked += hr[r] * 32.0 * u;
          }
        }
      }
      tasks = walked > 0.0 && useful / walked >= 0.35;
    }
  }
  // choose the number of CTAs that share a group: by default the fewest that hold one codeword
  // (an attention read of a key held by another CTA of the cluster costs far more than the
  // token rows left idle by a looser packing), with as many words per group as fit; an explicit
  // cluster_ctas is honoured when it can hold a word
  int best_C = 0, best_G = 0;
  const int cmin = (T + kRows - 1) / kRows;
  for (int C = cmin; C <= kMaxCluster && !best_C; ++C) {
    if (tasks && C != 1) continue;
    if (d.cluster_ctas && C != d.cluster_ctas) continue;
    const int G = (tasks && D == 128) ? 1 : (C * kRows) / T;
    if (G < 1) continue;
    if (((G + C - 1) / C) * n > kOutBitsBytes) continue;
    best_C = C, best_G = G;
  }
  if (!best_C) return d.cluster_ctas ? AECCT_ERR_INVALID_ARG : AECCT_ERR_UNSUPPORTED;
  if (best_G * ((n + 31) / 32) > 128) return AECCT_ERR_UNSUPPORTED;  // hard-decision bitmasks of a group
  if (d.alpha_mode == 1 && best_C != 1) return AECCT_ERR_UNSUPPORTED;  // per-word alpha: one CTA per word

  // Per-row lists over per-head staged rows (d = 128): a head's K and V rows of the whole group
  // (128 bytes a row) are gathered into the 80 KB of the operand tile and the weight stages, and
  // each row's scores take TMEM columns [128, 384).  By default it replaces the per-row walk when
  // the group spans a cluster, where that walk reads every key through the distributed shared
  // memory window.
  size_t max_list = 0;
  for (int r = 0; r < 2; ++r)
    for (int t = 0; t < T; ++t) max_list = std::max(max_list, nb[r][t].size());
  const bool staged_ok = D == 128 && best_G * T <= kStagedMaxRows && max_list <= static_cast<size_t>(kStagedMaxKeys);
  int att = tasks ? 1 : 0;
  if (d.attention_mode == 3) {
    if (!staged_ok) return AECCT_ERR_UNSUPPORTED;
    att = 2;
  } else if (d.attention_mode == 0 && !tasks && staged_ok && best_C > 1) {
    att = 2;
  }

  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return AECCT_ERR_NO_DEVICE;
  cudaDeviceProp prop;
  e = cudaGetDeviceProperties(&prop, dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDeviceProperties");
  if (prop.major != 10) {
    g_last_error = "device is not compute capability 10.x";
    return AECCT_ERR_NO_DEVICE;
  }
  // a bound on the task plan's bytes (it sits in shared memory after the fixed regions)
  uint32_t plan_bound = 0;
  if (tasks) {
    const uint32_t ngb = D == 128 ? static_cast<uint32_t>((n + 31) / 32 + (m + 31) / 32)
                                  : static_cast<uint32_t>(best_G * ((T + 31) / 32));
    auto r16 = [](uint32_t v) { return (v + 15u) & ~15u; };
    plan_bound = r16(2u * kEpiWarps * kMaxTasks) + 16u * ngb +
                 r16(8u * ngb) + 2u * ngb * r16(static_cast<uint32_t>(T)) + 16u * 2u * 32u * ngb +
                 r16(4u + 8u * ngb);
    const uint32_t fixed = D == 32 ? SmemLayout<32, true>::kTotal
                           : D == 64 ? SmemLayout<64, true>::kTotal : SmemLayout<128, true>::kTotal;
    if (fixed + plan_bound > kMaxDynSmem) {
      g_last_error = "the warp-task plan does not fit shared memory";
      return AECCT_ERR_UNSUPPORTED;
    }
  }
  // staged mode with the cluster size left open: the size with the most words resident on the
  // device, words per group x clusters that fit at once (LDPC(128,64): three CTAs hold two words
  // in 46 clusters, 92 words, against 76 with two CTAs per word).  The group's rows stay within
  // the staged row limit.
  if (att == 2 && d.cluster_ctas == 0 && d.alpha_mode == 0) {
    int top = 0;
    for (int C = cmin; C <= kMaxCluster; ++C) {
      const int G = std::min(C * kRows / T, kStagedMaxRows / T);
      if (G < 1 || ((G + C - 1) / C) * n > kOutBitsBytes || G * ((n + 31) / 32) > 128) continue;
      int mc = 0;
      e = prepare_variant(d.activation, d.linear_mode, D, att, C, plan_bound, &mc);
      if (e != cudaSuccess) return cuda_fail(e, "kernel occupancy");
      if (G * mc > top) top = G * mc, best_C = C, best_G = G;
    }
  }
  int max_clusters = 0;
  e = prepare_variant(d.activation, d.linear_mode, D, att, best_C, plan_bound, &max_clusters);
  if (e != cudaSuccess) return cuda_fail(e, "kernel occupancy");
  if (max_clusters < 1) {
    g_last_error = "no cluster of this size fits on the device";
    return AECCT_ERR_UNSUPPORTED;
  }

  aecct_handle *h = new aecct_handle();
  h->n = n, h->k = k, h->T = T, h->m = m, h->d = D, h->n_layers = d.n_layers, h->h_first = d.h_first;
  h->Tp = (tasks && D == 128) ? Tp128 : T;
  h->d_spe = d.d_spe, h->C = best_C, h->G = best_G, h->max_clusters = max_clusters, h->att = att;
  h->ln_eps = d.ln_eps, h->alpha_floor = d.alpha_floor, h->b_d1 = d.b_d1, h->device = dev;
  h->alpha_mode = d.alpha_mode;
  h->activation = d.activation;
  h->linear_mode = d.linear_mode;
  h->att_scale = static_cast<float>(1.4426950408889634074 / std::sqrt(static_cast<double>(D / kHeads)));
  h->wait_limit = d.wait_limit_cycles ? d.wait_limit_cycles : (1LL << 32);

  // ---- H rows as bitmasks over the variables, for the syndromes (parity of popcounts)
  h->hwords = (n + 31) / 32;
  std::vector<uint32_t> hbits((size_t)m * h->hwords, 0u);
  for (int i = 0; i < m; ++i)
    for (int j = 0; j < n; ++j)
      if (d.H[(size_t)i * n + j]) hbits[(size_t)i * h->hwords + j / 32] |= 1u << (j % 32);
  // Rows of a codeword hold its tokens sorted by attention work (keys over the thread's first-ring
  // and second-ring head), so the 32 rows of a warp loop over similar key counts.
  std::vector<uint16_t> perm(h->Tp, 0xFFFFu), pos(T);
  if (tasks && D == 128) {
    // variables in rows 0..n-1, checks from the 32-row boundary npad; rows n..npad-1 hold no token
    for (int t = 0; t < T; ++t) {
      const int row = t < n ? t : npad + (t - n);
      perm[row] = static_cast<uint16_t>(t);
      pos[t] = static_cast<uint16_t>(row);
    }
  } else {
    std::vector<int> order(T);
    for (int t = 0; t < T; ++t) order[t] = t;
    const int hf = d.h_first, hs = d.heads - d.h_first;
    auto work = [&](int t) {
      const size_t a = hf > 0 ? nb[0][t].size() : 0, b = hs > 0 ? nb[1][t].size() : 0;
      return (hf > 0 && hs > 0) ? a + b : (a + b) * 2;
    };
    // task mode keeps the natural order (variables, then checks): query groups of one node type
    // share most of their keys
    if (!tasks) std::stable_sort(order.begin(), order.end(), [&](int a, int b) { return work(a) > work(b); });
    for (int i = 0; i < T; ++i) {
      perm[i] = static_cast<uint16_t>(order[i]);
      pos[order[i]] = static_cast<uint16_t>(i);
    }
  }
  // lists of row offsets, each padded to a multiple of 8 entries (one 16-byte load per 8 keys)
  std::vector<uint32_t> minfo[2];
  std::vector<uint16_t> mlist[2];
  for (int mk = 0; mk < 2; ++mk) {
    minfo[mk].assign(T, 0);
    for (int t = 0; t < T; ++t) {
      const size_t start = mlist[mk].size() / 8;
      const size_t cnt = nb[mk][t].size();
      if (cnt >= 2048 || start >= (1u << 21)) {
        g_last_error = "neighbour list too long";
        return AECCT_ERR_UNSUPPORTED;
      }
      minfo[mk][t] = static_cast<uint32_t>((start << 11) | cnt);
      for (uint16_t u : nb[mk][t]) mlist[mk].push_back(pos[u]);
      while (mlist[mk].size() % 8) mlist[mk].push_back(0);
    }
    if (mlist[mk].empty()) mlist[mk].assign(8, 0);
  }

  // ---- task-mode attention plan (every CTA holds the same layout: G codewords of T rows)
  std::vector<uint16_t> ptask;
  std::vector<uint32_t> pgrp, puinfo, pmask;
  std::vector<uint8_t> pqslot;
  std::vector<uint8_t> pulist;
  if (tasks) {
    const int G = best_G;
    struct Grp {
      int row0, lanes, cwrow0;
    };
    std::vector<Grp> grps;
    if (D == 128) {
      // one codeword; groups of the variables' rows, then of the checks' rows from npad: every group
      // starts on a lane quadrant (its padding rows, if any, come last)
      for (int off0 = 0; off0 < n; off0 += 32) grps.push_back({off0, std::min(32, n - off0), 0});
      for (int off0 = npad; off0 < h->Tp; off0 += 32) grps.push_back({off0, std::min(32, h->Tp - off0), 0});
    } else {
      for (int cw = 0; cw < G; ++cw)
        for (int off0 = 0; off0 < T; off0 += 32) grps.push_back({cw * T + off0, std::min(32, T - off0), cw * T});
    }
    const int ng = static_cast<int>(grps.size());
    std::vector<int> ucount(ng * 2, 0);
    pgrp.assign((size_t)ng * 4, 0);
    puinfo.assign((size_t)ng * 2, 0);
    pmask.assign((size_t)ng * 2 * 32 * 4, 0);
    for (int gi = 0; gi < ng; ++gi) {
      pgrp[gi * 4 + 0] = static_cast<uint32_t>(grps[gi].row0);
      pgrp[gi * 4 + 1] = static_cast<uint32_t>(grps[gi].lanes);
      pgrp[gi * 4 + 2] = static_cast<uint32_t>(grps[gi].cwrow0);
      const int off0 = grps[gi].row0 - grps[gi].cwrow0;
      for (int ring = 0; ring < 2; ++ring) {
        // union of the lanes' key sets, in ascending token order
        std::vector<uint8_t> in(T, 0);
        for (int ln = 0; ln < grps[gi].lanes; ++ln)
          for (uint16_t u : nb[ring][perm[off0 + ln]]) in[u] = 1;
        std::vector<int> uni;
        for (int u = 0; u < T; ++u)
          if (in[u]) uni.push_back(u);
        const size_t start = pulist.size() / 16;
        puinfo[gi * 2 + ring] = static_cast<uint32_t>((start << 8) | uni.size());
        ucount[gi * 2 + ring] = static_cast<int>(uni.size());
        for (int u : uni) pulist.push_back(static_cast<uint8_t>(pos[u]));
        while (pulist.size() % 16) pulist.push_back(0);
        for (int ln = 0; ln < grps[gi].lanes; ++ln) {
          std::vector<uint8_t> mine(T, 0);
          for (uint16_t u : nb[ring][perm[off0 + ln]]) mine[u] = 1;
          for (size_t kk = 0; kk < uni.size(); ++kk)
            if (mine[uni[kk]]) pmask[((size_t)(gi * 2 + ring) * 32 + ln) * 4 + kk / 32] |= 1u << (kk % 32);
        }
      }
    }
    // tasks (group, head), longest first.  d = 128: each on a warp of its group's TMEM lane quadrant,
    // where its rows' Q and A live (warps w with w % 4 = quadrant: one scheduler); d <= 64: the
    // schedulers by longest first onto the least-loaded one.  Then the warps of each scheduler by
    // assign_scheduler.
    std::vector<std::pair<int, int>> tl;  // (cost, task)
    for (int gi = 0; gi < ng; ++gi)
      for (int e = 0; e < kHeads; ++e) tl.push_back({ucount[gi * 2 + (e < d.h_first ? 0 : 1)] + 4, gi * 8 + e});
    std::stable_sort(tl.begin(), tl.end(), [](const std::pair<int, int> &x, const std::pair<int, int> &y) {
      return x.first > y.first;
    });
    std::vector<std::pair<int, int>> per_sched[4];
    long sched_load[4] = {0, 0, 0, 0};
    for (const auto &tk : tl) {
      int q = 0;
      if (D == 128) {
        q = (grps[tk.second / 8].row0 / 32) & 3;
      } else {
        for (int c = 1; c < 4; ++c)
          if (sched_load[c] < sched_load[q]) q = c;
      }
      per_sched[q].push_back(tk);
      sched_load[q] += tk.first;
    }
    // d = 128: a task may also run on a warp of a scheduler whose lane quadrant holds no token row,
    // its Q and A then in a 2 KB slot of weight stage W2 (idle from the previous block's FFN2 to this
    // block's O GEMM) instead of its rows' TMEM lanes.  Every loaded scheduler hands over the subset
    // of its tasks (at most kQSlots in all) whose cost comes closest to its excess over the mean load
    // without passing it; each goes to the free scheduler with the least load.  BCH(63,36): the fourth
    // quadrant holds no token row, and each of the other three hands it a 67 and a 31 (all at 294).
    std::vector<uint8_t> slot_of((size_t)ng * 8, 0xFFu);
    if (D == 128) {
      auto by_cost = [](const std::pair<int, int> &x, const std::pair<int, int> &y) { return x.first > y.first; };
      std::vector<int> free_q;
      long total = 0;
      for (int q = 0; q < 4; ++q) {
        total += sched_load[q];
        if (per_sched[q].empty()) free_q.push_back(q);
      }
      const long mean = total / 4;
      int nmoved = 0;
      for (int pass = 0; pass < 4 && !free_q.empty(); ++pass) {
        int q = -1;  // the most loaded scheduler not handled yet
        for (int c = 0; c < 4; ++c)
          if (!per_sched[c].empty() && std::find(free_q.begin(), free_q.end(), c) == free_q.end() &&
              sched_load[c] > mean && (q < 0 || sched_load[c] > sched_load[q]))
            q = c;
        if (q < 0) break;
        const long excess = sched_load[q] - mean;
        const int mt = static_cast<int>(std::min<size_t>(per_sched[q].size(), 12));
        uint32_t best_set = 0;
        long best_sum = 0;
        for (uint32_t set = 1; set < (1u << mt); ++set) {
          const int k = __builtin_popcount(set);
          if (nmoved + k > kQSlots) continue;
          long sum = 0;
          for (int t = 0; t < mt; ++t)
            if (set >> t & 1u) sum += per_sched[q][t].first;
          if (sum <= excess && (sum > best_sum || (sum == best_sum && k < __builtin_popcount(best_set))))
            best_sum = sum, best_set = set;
        }
        for (int t = mt - 1; t >= 0; --t) {
          if (!(best_set >> t & 1u)) continue;
          int fq = free_q[0];
          for (int c : free_q)
            if (sched_load[c] < sched_load[fq]) fq = c;
          const std::pair<int, int> tk = per_sched[q][t];
          per_sched[q].erase(per_sched[q].begin() + t);
          sched_load[q] -= tk.first;
          per_sched[fq].push_back(tk);
          sched_load[fq] += tk.first;
          slot_of[tk.second] = static_cast<uint8_t>(nmoved++);
        }
        sched_load[q] = std::min(sched_load[q], mean);  // handled: not picked again
      }
      for (int q = 0; q < 4; ++q) std::stable_sort(per_sched[q].begin(), per_sched[q].end(), by_cost);
      // the group of each lane quadrant (every group of a d = 128 word starts on one), then the slots
      pqslot.assign(4 + (size_t)ng * 8, 0xFFu);
      for (int gi = 0; gi < ng; ++gi) pqslot[(grps[gi].row0 / 32) & 3] = static_cast<uint8_t>(gi);
      std::copy(slot_of.begin(), slot_of.end(), pqslot.begin() + 4);
    }
    ptask.assign((size_t)kEpiWarps * kMaxTasks, 0xFFFFu);
    for (int q = 0; q < 4; ++q) {
      std::vector<int> cost, slot;
      for (const auto &tk : per_sched[q]) cost.push_back(tk.first);
      if (!assign_scheduler(cost, kMaxTasks, slot)) {
        free_handle(h);
        g_last_error = "attention plan: too many tasks for a warp";
        return AECCT_ERR_UNSUPPORTED;
      }
      int cnt[4] = {0, 0, 0, 0};
      for (size_t i = 0; i < per_sched[q].size(); ++i) {
        const int w = q + 4 * slot[i];
        ptask[(size_t)w * kMaxTasks + cnt[slot[i]]++] = static_cast<uint16_t>(per_sched[q][i].second);
      }
    }
  }

  // ---- weights: 2-bit codes (or full-precision values rounded to bf16) -> bf16 K-major
  // core-matrix chunks, in the order the MMA consumes them
  const Gemm gemms[4] = {{3 * D, D}, {D, D}, {F, D}, {D, F}};
  const int nch = schedule_chunks(D, h->chunks);
  const uint32_t off = h->chunks[nch - 1].off + h->chunks[nch - 1].bytes;
  h->n_chunks = nch;
  h->layer_bytes = off;
  // AAP linears: the 2-bit codes go to the device as they are and a kernel expands them there
  // (aap.cu, unpack_weights_kernel); full-precision linears are rounded to bf16 and laid out here
  const bool gpu_unpack = d.linear_mode == 0;
  std::vector<uint16_t> ws(gpu_unpack ? 0 : (size_t)d.n_layers * off / 2, 0);
  if (!gpu_unpack) {
    const size_t per_layer_packed = 12u * (size_t)D * D / 4u, per_layer_full = 12u * (size_t)D * D;
    std::vector<uint16_t> W[4];  // bf16 encodings, [N][K] per GEMM
    for (int l = 0; l < d.n_layers; ++l) {
      // the six matrices in ABI order, as bf16: ternary codes unpacked (exact), or
      // full-precision values rounded to nearest even
      auto unpack = [&](size_t first, int rows, int cols, uint16_t *dst) {
        if (d.linear_mode == 0) {
          const uint8_t *src = d.w_packed + per_layer_packed * l + first / 4;
          for (int r = 0; r < rows; ++r)
            for (int c = 0; c < cols; ++c) {
              const uint8_t byte = src[(size_t)r * (cols / 4) + c / 4];
              dst[(size_t)r * cols + c] = f2bf_bits(static_cast<float>(tern((byte >> (2 * (c % 4))) & 3u)));
            }
        } else {
          const float *src = d.w_full + per_layer_full * l + first;
          for (size_t i = 0; i < (size_t)rows * cols; ++i) dst[i] = bf16_rne_bits(src[i]);
        }
      };
      for (int g = 0; g < 4; ++g) W[g].assign((size_t)gemms[g].N * gemms[g].K, 0);
      const size_t dd = (size_t)D * D;
      unpack(0, D, D, W[0].data());                        // W_q -> QKV rows [0, D)
      unpack(dd, D, D, W[0].data() + dd);                  // W_k -> rows [D, 2D)
      unpack(2 * dd, D, D, W[0].data() + 2 * dd);          // W_v -> rows [2D, 3D)
      unpack(3 * dd, D, D, W[1].data());                   // W_o
      unpack(4 * dd, F, D, W[2].data());                   // W_1
      unpack(4 * dd + (size_t)F * D, D, F, W[3].data());   // W_2
      uint16_t *lw = ws.data() + (size_t)l * off / 2;
      for (int c = 0; c < nch; ++c) {
        const ChunkDesc &ch = h->chunks[c];
        const Gemm gm = gemms[ch.gemm];
        uint8_t *base = reinterpret_cast<uint8_t *>(lw) + ch.off;
        for (int rr = 0; rr < ch.nrows; ++rr)
          for (int cc = 0; cc < ch.kcols; ++cc) {
            // FFN1's output column n0 + rr holds hidden unit ffn1_unit_of_column (d = 128)
            const int row = ch.gemm == 2 ? ffn1_unit_of_column(D, ch.n0 + rr) : ch.n0 + rr;
            const uint16_t bits = W[ch.gemm][(size_t)row * gm.K + ch.k0 + cc];
            std::memcpy(base + core_off(rr, cc, ch.kcols), &bits, 2);
          }
      }
    }
  }
  // ---- per-block parameter vectors
  const int LPS = LayerParamLayout::stride(D);
  std::vector<float> lpv((size_t)d.n_layers * LPS, 0.0f);
  for (int l = 0; l < d.n_layers; ++l) {
    float *v = lpv.data() + (size_t)l * LPS;
    std::memcpy(v, d.bias + (size_t)l * 9 * D, sizeof(float) * 9 * D);  // b_q b_k b_v b_o b_1 b_2
    std::memcpy(v + LayerParamLayout::ln1g(D), d.ln_gamma + (size_t)l * 2 * D, sizeof(float) * D);
    std::memcpy(v + LayerParamLayout::ln1b(D), d.ln_beta + (size_t)l * 2 * D, sizeof(float) * D);
    std::memcpy(v + LayerParamLayout::ln2g(D), d.ln_gamma + (size_t)l * 2 * D + D, sizeof(float) * D);
    std::memcpy(v + LayerParamLayout::ln2b(D), d.ln_beta + (size_t)l * 2 * D + D, sizeof(float) * D);
    if (d.linear_mode == 0) std::memcpy(v + LayerParamLayout::sw(D), d.w_scale + (size_t)l * 6, sizeof(float) * 6);
    else for (int i = 0; i < 6; ++i) v[LayerParamLayout::sw(D) + i] = 1.0f;
  }
  // the task plan as one blob, each part on a 16-byte boundary
  std::vector<uint8_t> blob;
  if (tasks) {
    auto put = [&](const void *src, size_t bytes) {
      const uint32_t off = static_cast<uint32_t>(blob.size());
      blob.insert(blob.end(), static_cast<const uint8_t *>(src), static_cast<const uint8_t *>(src) + bytes);
      while (blob.size() % 16) blob.push_back(0);
      return off;
    };
    h->off_task = put(ptask.data(), ptask.size() * 2);
    h->off_grp = put(pgrp.data(), pgrp.size() * 4);
    h->off_uinfo = put(puinfo.data(), puinfo.size() * 4);
    h->off_ulist = put(pulist.data(), pulist.size());
    h->off_mask = put(pmask.data(), pmask.size() * 4);
    h->off_qslot = put(pqslot.data(), pqslot.size());
    h->plan_bytes = static_cast<uint32_t>(blob.size());
    if (h->plan_bytes > plan_bound) {
      free_handle(h);
      g_last_error = "internal: the task plan exceeds its bound";
      return AECCT_ERR_UNSUPPORTED;
    }
  }
  const int de = D - d.d_spe;
  if ((rc = dev_upload(h, &h->wstream, gpu_unpack ? nullptr : reinterpret_cast<const uint8_t *>(ws.data()),
                      (size_t)d.n_layers * off)) ||
      (rc = dev_upload(h, &h->lparams, lpv.data(), lpv.size())) ||
      (rc = dev_upload(h, &h->emb, d.emb, (size_t)T * de)) ||
      (rc = dev_upload(h, &h->spe, d.spe, (size_t)T * d.d_spe)) ||
      (rc = dev_upload(h, &h->w_d1, d.w_d1, (size_t)D)) ||
      (rc = dev_upload(h, &h->w_out, d.w_out, (size_t)T * n)) ||
      (rc = dev_upload(h, &h->b_out, d.b_out, (size_t)n)) ||
      (rc = dev_upload(h, &h->hbits, hbits.data(), hbits.size())) ||
      (rc = dev_upload(h, &h->perm, perm.data(), perm.size())) ||
      (rc = dev_upload(h, &h->pos, pos.data(), pos.size())) ||
      (rc = dev_upload(h, &h->mask_info[0], minfo[0].data(), minfo[0].size())) ||
      (rc = dev_upload(h, &h->mask_list[0], mlist[0].data(), mlist[0].size())) ||
      (rc = dev_upload(h, &h->mask_info[1], minfo[1].data(), minfo[1].size())) ||
      (rc = dev_upload(h, &h->mask_list[1], mlist[1].data(), mlist[1].size())) ||
      (rc = dev_upload(h, &h->plan_blob, blob.data(), blob.size())) ||
      (rc = dev_upload<float>(h, &h->kv_scratch, nullptr,
                              att == 2 ? (size_t)max_clusters * best_C * kRows * kHeads * 2 * 16 : 1)) ||
      (rc = dev_upload<int>(h, &h->d_err, nullptr, 1))) {
    free_handle(h);
    return rc;
  }
  if (gpu_unpack) {
    uint8_t *packed = nullptr;
    const size_t pbytes = (size_t)d.n_layers * 3u * (size_t)D * D;
    if ((e = cudaMalloc(&packed, pbytes)) == cudaSuccess &&
        (e = cudaMemcpy(packed, d.w_packed, pbytes, cudaMemcpyHostToDevice)) == cudaSuccess &&
        (e = launch_unpack_weights(packed, d.n_layers, D, h->chunks, nch, off, h->wstream, nullptr)) == cudaSuccess)
      e = cudaDeviceSynchronize();
    cudaFree(packed);
    if (e != cudaSuccess) {
      free_handle(h);
      return cuda_fail(e, "weight unpack");
    }
  }
  if ((e = cudaMemset(h->d_err, 0, sizeof(int))) != cudaSuccess ||
      (e = cudaHostAlloc(reinterpret_cast<void **>(&h->h_err), sizeof(int), cudaHostAllocDefault)) != cudaSuccess ||
      (e = cudaEventCreateWithFlags(&h->ev, cudaEventDisableTiming)) != cudaSuccess) {
    free_handle(h);
    return cuda_fail(e, "create");
  }
  *h->h_err = 0;
  *out = h;
  return AECCT_OK;
}

// the kernel arguments of one decode call: the handle's model and plan, this call's buffers
static DecodeParams decode_params(const aecct_handle *h, int64_t B, const float *y_dev, uint8_t *bits_dev,
                                  uint8_t *syn_dev, float *logits_dev, int *err_dev) {
  DecodeParams p = {};
  p.n = h->n, p.k = h->k, p.T = h->T, p.m = h->m, p.n_layers = h->n_layers, p.h_first = h->h_first;
  p.Tp = h->Tp;
  p.d_spe = h->d_spe, p.C = h->C, p.G = h->G;
  p.B = B;
  p.n_groups = (B + h->G - 1) / h->G;
  p.n_clusters = static_cast<int>(p.n_groups < h->max_clusters ? p.n_groups : h->max_clusters);
  p.y = y_dev, p.bits = bits_dev, p.syn = syn_dev, p.logits = logits_dev;
  p.wstream = h->wstream, p.layer_bytes = h->layer_bytes;
  p.lparams = h->lparams, p.emb = h->emb, p.spe = h->spe, p.w_d1 = h->w_d1, p.b_d1 = h->b_d1;
  p.w_out = h->w_out, p.b_out = h->b_out, p.hbits = h->hbits, p.hwords = h->hwords;
  p.perm = h->perm, p.pos = h->pos;
  p.plan_blob = reinterpret_cast<const uint4 *>(h->plan_blob), p.plan_bytes = h->plan_bytes;
  p.off_task = h->off_task, p.off_grp = h->off_grp;
  p.off_uinfo = h->off_uinfo, p.off_ulist = h->off_ulist, p.off_mask = h->off_mask, p.off_qslot = h->off_qslot;
  p.mask_info[0] = h->mask_info[0], p.mask_info[1] = h->mask_info[1];
  p.mask_list[0] = reinterpret_cast<const uint4 *>(h->mask_list[0]);
  p.mask_list[1] = reinterpret_cast<const uint4 *>(h->mask_list[1]);
  p.ln_eps = h->ln_eps, p.alpha_floor = h->alpha_floor, p.att_scale = h->att_scale, p.alpha_mode = h->alpha_mode;
  p.cap_B = h->cap_B, p.cap_q = h->cap_q, p.cap_acc = h->cap_acc, p.cap_alpha = h->cap_alpha, p.cap_syn = h->cap_syn;
  p.kv_scratch = h->kv_scratch;
  p.err = err_dev, p.wait_limit = h->wait_limit;
  return p;
}

// The handle's model, plan and status word live on the device that was current at create; a
// decode launched while another device is current would read them from the wrong GPU.
static int check_device(const aecct_handle *h, const char *who) {
  int dev = -1;
  const cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  if (dev != h->device) {
    g_last_error = std::string(who) + ": the current device is " + std::to_string(dev) +
                   ", the handle was created on device " + std::to_string(h->device);
    return AECCT_ERR_INVALID_ARG;
  }
  return AECCT_OK;
}

static int collect_status(aecct_handle *h, bool block) {
  if (!h->ev_pending) {
    const int s = h->pending_status;
    h->pending_status = AECCT_OK;
    return s;
  }
  cudaError_t e = block ? cudaEventSynchronize(h->ev) : cudaEventQuery(h->ev);
  if (e == cudaErrorNotReady) return AECCT_OK;
  h->ev_pending = false;
  if (e != cudaSuccess) return cuda_fail(e, "decode kernel");
  if (*h->h_err) {
    *h->h_err = 0;
    cudaMemset(h->d_err, 0, sizeof(int));
    g_last_error = "a device-side wait exceeded its limit";
    return AECCT_ERR_TIMEOUT;
  }
  return AECCT_OK;
}

int aecct_decode(aecct_handle *h, const float *y_dev, int64_t B, uint8_t *bits_dev, uint8_t *syndrome_dev,
                 float *logits_dev, void *cuda_stream) {
  if (!h || B < 0) return AECCT_ERR_INVALID_ARG;
  if (B == 0) return AECCT_OK;
  if (!y_dev || !bits_dev) return AECCT_ERR_INVALID_ARG;
  if (const int rc = check_device(h, "aecct_decode")) return rc;
  cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);
  const int prev = collect_status(h, false);
  if (prev != AECCT_OK) return prev;
  const DecodeParams p = decode_params(h, B, y_dev, bits_dev, syndrome_dev, logits_dev, h->d_err);
  cudaError_t e;
  e = launch_variant(h->activation, h->linear_mode, h->d, h->att, p, stream);
  if (e != cudaSuccess) return cuda_fail(e, "decode launch");
  if ((e = cudaMemcpyAsync(h->h_err, h->d_err, sizeof(int), cudaMemcpyDeviceToHost, stream)) != cudaSuccess)
    return cuda_fail(e, "status copy");
  if ((e = cudaEventRecord(h->ev, stream)) != cudaSuccess) return cuda_fail(e, "event record");
  h->ev_pending = true;
  return AECCT_OK;
}

int aecct_synchronize(aecct_handle *h) {
  if (!h) return AECCT_ERR_INVALID_ARG;
  return collect_status(h, true);
}

int aecct_decode_host(aecct_handle *h, const float *y_host, int64_t B, uint8_t *bits_host, uint8_t *syndrome_host,
                      float *logits_host, void *cuda_stream) {
  if (!h || B < 0) return AECCT_ERR_INVALID_ARG;
  if (B == 0) return AECCT_OK;
  if (!y_host || !bits_host) return AECCT_ERR_INVALID_ARG;
  if (const int rc = check_device(h, "aecct_decode_host")) return rc;
  cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);
  cudaError_t e;
  if (B > h->stage_B) {
    cudaFree(h->st_y), cudaFree(h->st_bits), cudaFree(h->st_syn), cudaFree(h->st_logits);
    h->st_y = nullptr, h->st_bits = nullptr, h->st_syn = nullptr, h->st_logits = nullptr, h->stage_B = 0;
    if ((e = cudaMalloc(&h->st_y, sizeof(float) * B * h->n)) != cudaSuccess ||
        (e = cudaMalloc(&h->st_bits, (size_t)B * h->n)) != cudaSuccess ||
        (e = cudaMalloc(&h->st_syn, (size_t)B * h->m)) != cudaSuccess ||
        (e = cudaMalloc(&h->st_logits, sizeof(float) * B * h->n)) != cudaSuccess)
      return e == cudaErrorMemoryAllocation ? AECCT_ERR_OUT_OF_MEMORY : cuda_fail(e, "staging");
    h->stage_B = B;
  }
  if ((e = cudaMemcpyAsync(h->st_y, y_host, sizeof(float) * B * h->n, cudaMemcpyHostToDevice, stream)) != cudaSuccess)
    return cuda_fail(e, "copy y");
  int rc = aecct_decode(h, h->st_y, B, h->st_bits, syndrome_host ? h->st_syn : nullptr,
                        logits_host ? h->st_logits : nullptr, cuda_stream);
  if (rc) return rc;
  if ((e = cudaMemcpyAsync(bits_host, h->st_bits, (size_t)B * h->n, cudaMemcpyDeviceToHost, stream)) != cudaSuccess)
    return cuda_fail(e, "copy bits");
  if (syndrome_host &&
      (e = cudaMemcpyAsync(syndrome_host, h->st_syn, (size_t)B * h->m, cudaMemcpyDeviceToHost, stream)) != cudaSuccess)
    return cuda_fail(e, "copy syndrome");
  if (logits_host && (e = cudaMemcpyAsync(logits_host, h->st_logits, sizeof(float) * B * h->n,
                                          cudaMemcpyDeviceToHost, stream)) != cudaSuccess)
    return cuda_fail(e, "copy logits");
  if ((e = cudaStreamSynchronize(stream)) != cudaSuccess) return cuda_fail(e, "stream sync");
  return collect_status(h, true);
}

// ---- host-buffer decode with no allocation (the paper has no counterpart).  Callers that must
// not allocate device memory while they decode -- a fixed device-memory budget taken up front,
// or a latency-bound loop where cudaMalloc/cudaFree may synchronise the device -- get their
// staging and the kernel's status word from this static array instead of cudaMalloc.
namespace {
__device__ __align__(256) unsigned char g_noalloc_scratch[AECCT_NOALLOC_SCRATCH_BYTES];
constexpr int kNoAllocMaxDevices = 64;
void *g_noalloc_base[kNoAllocMaxDevices] = {};  // per device, resolved by its first call
size_t round256(size_t v) { return (v + 255u) & ~static_cast<size_t>(255u); }
}  // namespace

int aecct_decode_host_noalloc(aecct_handle *h, const float *y_host, int64_t B, uint8_t *bits_host,
                              uint8_t *syndrome_host, float *logits_host, void *cuda_stream) {
  if (!h || B < 0) return AECCT_ERR_INVALID_ARG;
  if (B == 0) return AECCT_OK;
  if (!y_host || !bits_host) return AECCT_ERR_INVALID_ARG;
  // the scratch used is the current device's, so the current device must be the handle's
  if (const int rc = check_device(h, "aecct_decode_host_noalloc")) return rc;
  // an earlier asynchronous aecct_decode on this handle reports its status first, as in
  // aecct_decode
  if (const int prev = collect_status(h, false)) return prev;
  const int dev = h->device;
  cudaError_t e;
  if (dev < 0 || dev >= kNoAllocMaxDevices) {
    g_last_error = "aecct_decode_host_noalloc: device index beyond the per-device table";
    return AECCT_ERR_UNSUPPORTED;
  }
  if (!g_noalloc_base[dev]) {  // set-up, once per device, with that device current
    void *base = nullptr;
    if ((e = cudaGetSymbolAddress(&base, g_noalloc_scratch)) != cudaSuccess)
      return cuda_fail(e, "cudaGetSymbolAddress (aecct_decode_host_noalloc scratch)");
    g_noalloc_base[dev] = base;
  }
  // layout: status word | y | bits | syndromes | logits, each part on a 256-byte boundary.  A word
  // takes at least 5n bytes (y and bits), so a B beyond scratch / 5n is refused before any size
  // product is formed (no size_t wrap-around for huge B).
  const size_t n = static_cast<size_t>(h->n), m = static_cast<size_t>(h->m);
  if (static_cast<uint64_t>(B) > AECCT_NOALLOC_SCRATCH_BYTES / (5u * n)) {
    g_last_error = "aecct_decode_host_noalloc: B = " + std::to_string(B) + " words need more than the " +
                   std::to_string(AECCT_NOALLOC_SCRATCH_BYTES) + "-byte static scratch holds";
    return AECCT_ERR_INVALID_ARG;
  }
  const size_t b = static_cast<size_t>(B);
  const size_t off_y = 256, off_bits = off_y + round256(sizeof(float) * b * n), off_syn = off_bits + round256(b * n);
  const size_t off_log = off_syn + (syndrome_host ? round256(b * m) : 0);
  const size_t end = off_log + (logits_host ? round256(sizeof(float) * b * n) : 0);
  if (end > AECCT_NOALLOC_SCRATCH_BYTES) {
    g_last_error = "aecct_decode_host_noalloc: B = " + std::to_string(B) + " needs " + std::to_string(end) +
                   " bytes of staging, more than the " + std::to_string(AECCT_NOALLOC_SCRATCH_BYTES) +
                   "-byte static scratch holds";
    return AECCT_ERR_INVALID_ARG;
  }
  uint8_t *base = static_cast<uint8_t *>(g_noalloc_base[dev]);
  int *err = reinterpret_cast<int *>(base);
  float *y_dev = reinterpret_cast<float *>(base + off_y);
  uint8_t *bits_dev = base + off_bits;
  uint8_t *syn_dev = syndrome_host ? base + off_syn : nullptr;
  float *logits_dev = logits_host ? reinterpret_cast<float *>(base + off_log) : nullptr;
  cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);
  // the status word must start at zero (the kernel only ORs into it)
  if ((e = cudaMemsetAsync(err, 0, sizeof(int), stream)) != cudaSuccess) return cuda_fail(e, "clear status");
  if ((e = cudaMemcpyAsync(y_dev, y_host, sizeof(float) * b * n, cudaMemcpyHostToDevice, stream)) != cudaSuccess)
    return cuda_fail(e, "copy y");
  const DecodeParams p = decode_params(h, B, y_dev, bits_dev, syn_dev, logits_dev, err);
  e = launch_variant(h->activation, h->linear_mode, h->d, h->att, p, stream);
  if (e != cudaSuccess) return cuda_fail(e, "decode launch");
  if ((e = cudaMemcpyAsync(bits_host, bits_dev, b * n, cudaMemcpyDeviceToHost, stream)) != cudaSuccess)
    return cuda_fail(e, "copy bits");
  if (syndrome_host && (e = cudaMemcpyAsync(syndrome_host, syn_dev, b * m, cudaMemcpyDeviceToHost, stream)) != cudaSuccess)
    return cuda_fail(e, "copy syndrome");
  if (logits_host &&
      (e = cudaMemcpyAsync(logits_host, logits_dev, sizeof(float) * b * n, cudaMemcpyDeviceToHost, stream)) != cudaSuccess)
    return cuda_fail(e, "copy logits");
  int status_word = 0;
  if ((e = cudaMemcpyAsync(&status_word, err, sizeof(int), cudaMemcpyDeviceToHost, stream)) != cudaSuccess)
    return cuda_fail(e, "copy status");
  if ((e = cudaStreamSynchronize(stream)) != cudaSuccess) return cuda_fail(e, "stream sync");
  if (status_word) {
    g_last_error = "a device-side wait exceeded its limit";
    return AECCT_ERR_TIMEOUT;
  }
  return AECCT_OK;
}

int aecct_set_capture(aecct_handle *h, int64_t cap_B, int8_t *q_dev, int32_t *acc_dev, float *alpha_dev,
                      uint8_t *syn_dev) {
  if (!h || cap_B < 0) return AECCT_ERR_INVALID_ARG;
  h->cap_B = cap_B;
  h->cap_q = cap_B ? q_dev : nullptr;
  h->cap_acc = cap_B ? acc_dev : nullptr;
  h->cap_alpha = cap_B ? alpha_dev : nullptr;
  h->cap_syn = cap_B ? syn_dev : nullptr;
  return AECCT_OK;
}

int aecct_query(const aecct_handle *h, int32_t *cluster_ctas, int32_t *words_per_group, int32_t *max_clusters,
                int32_t *threads_per_cta, int32_t *smem_bytes, int32_t *attention_mode) {
  if (!h) return AECCT_ERR_INVALID_ARG;
  if (cluster_ctas) *cluster_ctas = h->C;
  if (words_per_group) *words_per_group = h->G;
  if (max_clusters) *max_clusters = h->max_clusters;
  if (threads_per_cta) *threads_per_cta = kThreads;
  int sm;
  const bool tasks = h->att == 1;
  if (h->d == 32) sm = tasks ? SmemLayout<32, true>::kTotal : SmemLayout<32>::kTotal;
  else if (h->d == 64) sm = tasks ? SmemLayout<64, true>::kTotal : SmemLayout<64>::kTotal;
  else sm = tasks ? SmemLayout<128, true>::kTotal : SmemLayout<128>::kTotal;
  if (smem_bytes) *smem_bytes = sm + static_cast<int32_t>(h->plan_bytes);
  if (attention_mode) *attention_mode = h->att == 1 ? 2 : (h->att == 2 ? 3 : 1);
  return AECCT_OK;
}

int aecct_destroy(aecct_handle *h) {
  if (!h) return AECCT_ERR_INVALID_ARG;
  if (h->ev_pending) cudaEventSynchronize(h->ev);
  free_handle(h);
  return AECCT_OK;
}

int aecct_selftest_mma(const int8_t *a_host, const int8_t *b_host, int32_t K, int32_t N, float *out_host) {
  if (!a_host || !b_host || !out_host) return AECCT_ERR_INVALID_ARG;
  if (K < 16 || K > 128 || K % 16 || N < 16 || N > 256 || N % 16) return AECCT_ERR_INVALID_ARG;
  cudaError_t e = run_selftest_mma(a_host, b_host, K, N, out_host);
  if (e == cudaErrorTimeout) return AECCT_ERR_TIMEOUT;
  return e == cudaSuccess ? AECCT_OK : cuda_fail(e, "selftest mma");
}

int aecct_selftest_timeout(int64_t limit_cycles, int32_t *status_host) {
  if (!status_host || limit_cycles <= 0) return AECCT_ERR_INVALID_ARG;
  int st = -1;
  cudaError_t e = run_selftest_timeout(limit_cycles, &st);
  if (e != cudaSuccess) return cuda_fail(e, "selftest timeout");
  *status_host = st == 1 ? AECCT_ERR_TIMEOUT : (st == 0 ? AECCT_OK : AECCT_ERR_CUDA);
  return AECCT_OK;
}

int aecct_spe_table(const uint8_t *H, int32_t n, int32_t k, int32_t d_spe, int32_t heads, const double *w_pe,
                    const double *wq, const double *wk, const double *wv, const double *wo, float *spe_out,
                    double *lam_out, double *U_out, double *spe64_out) {
  if (!H || !w_pe || !wq || !wk || !wv || !wo || !spe_out) return AECCT_ERR_INVALID_ARG;
  if (n <= 0 || k <= 0 || k >= n || n + (n - k) > kSpeMaxTokens) return AECCT_ERR_INVALID_ARG;
  if (heads < 1 || heads > kSpeMaxHeads || d_spe < heads || d_spe % heads != 0) return AECCT_ERR_INVALID_ARG;
  const int m = n - k;
  for (size_t i = 0; i < static_cast<size_t>(m) * n; ++i)
    if (H[i] > 1) return AECCT_ERR_INVALID_ARG;
  int sweeps = 0, status = 0;
  const cudaError_t e = run_spe_table(H, n, m, d_spe, heads, w_pe, wq, wk, wv, wo, 1e-8, 1e-6, spe_out, lam_out, U_out,
                                      spe64_out, &sweeps, &status);
  if (e != cudaSuccess) return cuda_fail(e, "spe table");
  if (status) {
    g_last_error = "spe table: a cluster of equal eigenvalues did not yield a full canonical basis";
    return AECCT_ERR_UNSUPPORTED;
  }
  return AECCT_OK;
}

int aecct_aap_ternarize(const float *w_dev, int32_t n_tensors, const int64_t *len_host, const float *delta_host,
                        float eps, uint8_t *packed_dev, float *scale_dev, float *wq_dev, void *cuda_stream) {
  if (n_tensors < 0 || (n_tensors > 0 && (!w_dev || !len_host || !delta_host || !packed_dev || !scale_dev)))
    return AECCT_ERR_INVALID_ARG;
  if (!(eps > 0.0f) || !std::isfinite(eps)) return AECCT_ERR_INVALID_ARG;
  for (int j = 0; j < n_tensors; ++j) {
    if (len_host[j] < 4 || len_host[j] % 4 != 0 || len_host[j] > (int64_t(1) << 31)) return AECCT_ERR_INVALID_ARG;
    if (!(delta_host[j] > 0.0f) || !std::isfinite(delta_host[j])) return AECCT_ERR_INVALID_ARG;
  }
  if (n_tensors == 0) return AECCT_OK;
  const cudaError_t e = launch_aap_ternarize(w_dev, n_tensors, len_host, delta_host, eps, packed_dev, scale_dev, wq_dev,
                                             static_cast<cudaStream_t>(cuda_stream));
  return e == cudaSuccess ? AECCT_OK : cuda_fail(e, "aap ternarize launch");
}

int aecct_selftest_fma_rate(int32_t paired, double *fma_per_s) {
  if (!fma_per_s || (paired != 0 && paired != 1)) return AECCT_ERR_INVALID_ARG;
  const cudaError_t e = run_selftest_fma_rate(paired != 0, fma_per_s);
  return e == cudaSuccess ? AECCT_OK : cuda_fail(e, "selftest fma rate");
}

}  // extern "C"
