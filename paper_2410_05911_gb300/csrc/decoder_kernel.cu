// decoder_kernel.cu -- the fused AECCT forward pass for sm_103a.
//
// One persistent kernel decodes the whole batch.  A cluster of C CTAs owns a group of G
// codewords whose T = 2n-k tokens are packed back to back over the cluster's C x 128 token
// rows (CTA c holds rows [128c, 128c + 128)).  Everything between the channel output y
// and the decoded bits stays on chip:
//
//   S1/S2  (Sec. 3, 4.3)   syndrome, tokens h(y), embedding + SPE       -> registers
//   S3-S8  (Sec. 4.1, 4.2, 5) per block:
//          Quant(x) -> tcgen05.mma QKV (bf16 operands holding exact int8 / ternary values,
//          fp32 accumulators in TMEM, exact integers) -> dequant -> K,V to shared memory
//          -> HPSA over CSR neighbour lists (DSMEM reads of peer CTAs) -> Quant(A) -> MMA O
//          -> dequant + residual + LayerNorm -> Quant -> MMA FFN1 -> dequant + ReLU ->
//          Quant -> MMA FFN2 -> dequant + residual + LayerNorm
//   S9/S10 (Sec. 3)        output head, hard decisions, syndrome of the decoded word
//
// Warp roles (576 threads): warps 0-15 do all CUDA-core work; thread (warp w, lane i) owns
// token row 32*(w%4) + i (the TMEM lane quadrant its warp may read) and column slice w/4;
// warp 16 streams weight chunks from global memory into a ring of shared-memory stages
// with the bulk-copy (TMA) engine; warp 17 issues the tensor-core MMAs.
//
// Every floating-point step uses one fixed order of IEEE fp32 operations (explicit _rn
// intrinsics, pairwise feature sums, two-pass base-2 softmax with a Taylor-series exp2), so
// the results are bit-identical to any implementation that follows the same order.
#include <cuda_runtime.h>

#include "aecct_internal.h"
#include "sm103_ptx.cuh"

namespace aecct {

// fp32(ln(2)^k / k!), k = 0..7: Taylor coefficients of 2^f = e^(f ln 2)
__device__ __forceinline__ float exp2_series(float x) {
  if (!(x >= -125.0f)) return 0.0f;
  const float n = rintf(x);
  const float f = __fsub_rn(x, n);
  float p = __uint_as_float(0x377fe5feu);      // k = 7
  p = __fmaf_rn(p, f, __uint_as_float(0x39218489u));  // k = 6
  p = __fmaf_rn(p, f, __uint_as_float(0x3aaec3ffu));  // k = 5
  p = __fmaf_rn(p, f, __uint_as_float(0x3c1d955bu));  // k = 4
  p = __fmaf_rn(p, f, __uint_as_float(0x3d635847u));  // k = 3
  p = __fmaf_rn(p, f, __uint_as_float(0x3e75fdf0u));  // k = 2
  p = __fmaf_rn(p, f, __uint_as_float(0x3f317218u));  // k = 1
  p = __fmaf_rn(p, f, 1.0f);                          // k = 0
  // p is in [0.70, 1.42] and n >= -125, so p * 2^n is normal: scale through the exponent field
  return __int_as_float(__float_as_int(p) + (static_cast<int>(n) << 23));
}

template <int N>
__device__ __forceinline__ float psum(const float *v) {
  if constexpr (N == 1) {
    return v[0];
  } else {
    return __fadd_rn(psum<N / 2>(v), psum<N / 2>(v + N / 2));
  }
}

struct Ctl {
  volatile int *abort;
  int *err;
  long long limit;
};

// Bounded mbarrier wait.  Returns false (and raises the CTA abort flag plus the device
// error word) when the phase does not complete within `limit` SM cycles; once the abort
// flag is up every later wait returns false at once so the kernel drains without blocking.
__device__ __noinline__ bool wait_bar(const Ctl &c, uint32_t bar, uint32_t parity, bool cluster_scope) {
  if (*c.abort) return false;
  if (cluster_scope ? mbar_try_wait_acq_cluster(bar, parity) : mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  while (true) {
    for (int i = 0; i < 32; ++i)
      if (cluster_scope ? mbar_try_wait_acq_cluster(bar, parity) : mbar_try_wait(bar, parity)) return true;
    if (*c.abort) return false;
    if (clock64() - t0 > c.limit) {
      *c.abort = 1;
      atomicOr(c.err, 1);
      return false;
    }
  }
}
// Teardown wait: ignores the abort flag (used to drain copies / MMAs in flight), still bounded.
__device__ __noinline__ bool wait_bar_drain(const Ctl &c, uint32_t bar, uint32_t parity) {
  const long long t0 = clock64();
  while (!mbar_try_wait(bar, parity)) {
    if (clock64() - t0 > c.limit) {
      atomicOr(c.err, 1);
      return false;
    }
  }
  return true;
}

// ------------------------------------------------------------------------------------------
// small helpers for the CUDA-core warps
// ------------------------------------------------------------------------------------------
__device__ __forceinline__ float q_code(float v, float r) {
  float q = rintf(__fmul_rn(v, r));
  q = q > 127.0f ? 127.0f : q;
  q = q < -127.0f ? -127.0f : q;
  return q;
}
__device__ __forceinline__ uint32_t pack_bf16x2(float a, float b) {
  // a, b are integers in [-127, 127]: exact in bf16
  __nv_bfloat162 v = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t *>(&v);
}
__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
  asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(a), "r"(b), "r"(c), "r"(d) : "memory");
}
__device__ __forceinline__ void st_shared_v2(uint32_t addr, uint32_t a, uint32_t b) {
  asm volatile("st.shared.v2.b32 [%0], {%1, %2};" ::"r"(addr), "r"(a), "r"(b) : "memory");
}
__device__ __forceinline__ void st_shared_f4(uint32_t addr, float a, float b, float c, float d) {
  asm volatile("st.shared.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "f"(a), "f"(b), "f"(c), "f"(d) : "memory");
}

// write the codes of LEN consecutive columns [c0, c0 + LEN) of row r into a K-major operand tile
// (c0 is a multiple of 8, or of 4 when LEN == 4)
template <int LEN>
__device__ __forceinline__ void store_codes(uint32_t tile, int r, int c0, int kdim, const float *q) {
  if constexpr (LEN == 4) {
    st_shared_v2(tile + core_off(r, c0, kdim), pack_bf16x2(q[0], q[1]), pack_bf16x2(q[2], q[3]));
  } else {
    static_assert(LEN % 8 == 0, "code run");
#pragma unroll
    for (int j = 0; j < LEN; j += 8)
      st_shared_v4(tile + core_off(r, c0 + j, kdim), pack_bf16x2(q[j], q[j + 1]), pack_bf16x2(q[j + 2], q[j + 3]),
                   pack_bf16x2(q[j + 4], q[j + 5]), pack_bf16x2(q[j + 6], q[j + 7]));
  }
}

template <int N>
__device__ __forceinline__ void ldg_vec(const float *src, float *dst) {
  static_assert(N % 4 == 0, "vector");
#pragma unroll
  for (int i = 0; i < N; i += 4) {
    const float4 v = __ldg(reinterpret_cast<const float4 *>(src + i));
    dst[i] = v.x;
    dst[i + 1] = v.y;
    dst[i + 2] = v.z;
    dst[i + 3] = v.w;
  }
}

// per-row reduction over the 4 column slices of a row: partial values go through shared memory
struct RowRed {
  float *buf;  // [2][4][128]
  int sel;
  __device__ __forceinline__ float *slot(int s, int r) { return buf + (sel * 4 + s) * kRows + r; }
};

// 16-bit entry k of an index block (k known at compile time after unrolling)
__device__ __forceinline__ int idx_at(const uint4 &w, int k) {
  const uint32_t word = k < 2 ? w.x : (k < 4 ? w.y : (k < 6 ? w.z : w.w));
  return static_cast<int>((k & 1) ? (word >> 16) : (word & 0xFFFFu));
}

// One (query, head) of HPSA (Sec. 4.2) over the neighbour rows described by `info` (see
// DecodeParams::mask_info).  Two passes in the canonical order:
// sigma_u = fma-chain(q . k_u) * scale, m = max sigma; p_u = 2^(sigma_u - m);
// l = sum p_u and num = sum p_u v_u in ascending key order; A = num * (1 / l).
// Keys come 8 per index load; U keys at a time have their loads issued together and their dot
// products run as independent chains, while every sum keeps the sequential key order.
template <int DH, int U, uint32_t STRIDE>
__device__ __forceinline__ void hpsa_head(const float *q, uint32_t info, const uint4 *__restrict__ lists,
                                          const uint64_t *kvgen, int rowbase, uint32_t hoff, float scale, float *A) {
  const uint4 *lst = lists + (info >> 11);
  const int cnt = static_cast<int>(info & 2047u);
  auto keyptr = [&](int off) -> const float4 * {
    const int ru = rowbase + off;
    return reinterpret_cast<const float4 *>(kvgen[ru >> 7] + static_cast<uint32_t>(ru & 127) * STRIDE + hoff);
  };
  auto dotk = [&](const float4 *kk) -> float {
    float dot = 0.0f;
#pragma unroll
    for (int i = 0; i < DH / 4; ++i) {
      dot = __fmaf_rn(q[4 * i], kk[i].x, dot);
      dot = __fmaf_rn(q[4 * i + 1], kk[i].y, dot);
      dot = __fmaf_rn(q[4 * i + 2], kk[i].z, dot);
      dot = __fmaf_rn(q[4 * i + 3], kk[i].w, dot);
    }
    return dot;
  };
  // pass 1: maximum score
  float mx = -INFINITY;
  for (int jb = 0; jb < cnt; jb += 8) {
    const uint4 w = __ldg(lst + (jb >> 3));
    if (jb + 8 <= cnt) {
#pragma unroll
      for (int k0 = 0; k0 < 8; k0 += U) {
        float4 kk[U][DH / 4];
#pragma unroll
        for (int k = 0; k < U; ++k) {
          const float4 *kp = keyptr(idx_at(w, k0 + k));
#pragma unroll
          for (int i = 0; i < DH / 4; ++i) kk[k][i] = kp[i];
        }
#pragma unroll
        for (int k = 0; k < U; ++k) mx = fmaxf(mx, __fmul_rn(dotk(kk[k]), scale));
      }
    } else {
      for (int k = 0; k < cnt - jb; ++k) {
        const float4 *kp = keyptr(idx_at(w, k));
        float4 kk[DH / 4];
#pragma unroll
        for (int i = 0; i < DH / 4; ++i) kk[i] = kp[i];
        mx = fmaxf(mx, __fmul_rn(dotk(kk), scale));
      }
    }
  }
  // pass 2: probabilities, their sum and the weighted values, in key order
  float lsum = 0.0f;
  float num[DH];
#pragma unroll
  for (int i = 0; i < DH; ++i) num[i] = 0.0f;
  auto accumulate = [&](float pr, const float4 *vv) {
    lsum = __fadd_rn(lsum, pr);
#pragma unroll
    for (int i = 0; i < DH / 4; ++i) {
      num[4 * i] = __fmaf_rn(pr, vv[i].x, num[4 * i]);
      num[4 * i + 1] = __fmaf_rn(pr, vv[i].y, num[4 * i + 1]);
      num[4 * i + 2] = __fmaf_rn(pr, vv[i].z, num[4 * i + 2]);
      num[4 * i + 3] = __fmaf_rn(pr, vv[i].w, num[4 * i + 3]);
    }
  };
  for (int jb = 0; jb < cnt; jb += 8) {
    const uint4 w = __ldg(lst + (jb >> 3));
    if (jb + 8 <= cnt) {
#pragma unroll
      for (int k0 = 0; k0 < 8; k0 += U) {
        float4 kk[U][DH / 4], vv[U][DH / 4];
#pragma unroll
        for (int k = 0; k < U; ++k) {
          const float4 *kp = keyptr(idx_at(w, k0 + k));
#pragma unroll
          for (int i = 0; i < DH / 4; ++i) kk[k][i] = kp[i];
#pragma unroll
          for (int i = 0; i < DH / 4; ++i) vv[k][i] = kp[DH / 4 + i];
        }
        float pr[U];
#pragma unroll
        for (int k = 0; k < U; ++k) pr[k] = exp2_series(__fsub_rn(__fmul_rn(dotk(kk[k]), scale), mx));
#pragma unroll
        for (int k = 0; k < U; ++k) accumulate(pr[k], vv[k]);
      }
    } else {
      for (int k = 0; k < cnt - jb; ++k) {
        const float4 *kp = keyptr(idx_at(w, k));
        float4 kk[DH / 4], vv[DH / 4];
#pragma unroll
        for (int i = 0; i < DH / 4; ++i) kk[i] = kp[i];
#pragma unroll
        for (int i = 0; i < DH / 4; ++i) vv[i] = kp[DH / 4 + i];
        accumulate(exp2_series(__fsub_rn(__fmul_rn(dotk(kk), scale), mx)), vv);
      }
    }
  }
  const float inv = __fdiv_rn(1.0f, lsum);
#pragma unroll
  for (int i = 0; i < DH; ++i) A[i] = __fmul_rn(num[i], inv);
}

// ------------------------------------------------------------------------------------------
// weight streaming and tensor-core issue (run by thread 0 of each CTA)
// ------------------------------------------------------------------------------------------
// Weight chunks are consumed in a fixed sequence: for each group of codewords, for each block,
// the block's chunks (QKV, then O, FFN1, FFN2).  Chunk i of the sequence uses ring stage i % S;
// its copy completes phase i / S of full[stage], its MMAs release phase i / S of empty[stage].
struct IssueState {
  int64_t total;   // chunks this CTA consumes
  int64_t issued;  // chunks whose copy has been started
  int64_t used;    // chunks whose MMAs have been issued
  uint32_t oph;    // parity of the next operand-ready phase
};

template <int D>
__device__ __noinline__ void issue_copies(const DecodeParams &p, const Ctl &ctl, IssueState &st, int64_t limit,
                                          uint32_t sb) {
  using L = SmemLayout<D>;
  constexpr int S = L::kStages;
  const uint32_t bar_full = sb + L::kOffBar, bar_empty = bar_full + 8 * S;
  if (limit > st.total) limit = st.total;
  while (st.issued < limit) {
    if (*ctl.abort) return;
    const int s = static_cast<int>(st.issued % S);
    if (st.issued >= S) wait_bar(ctl, bar_empty + 8 * s, static_cast<uint32_t>((st.issued / S - 1) & 1), false);
    const int c = static_cast<int>(st.issued % p.n_chunks);
    const int l = static_cast<int>((st.issued / p.n_chunks) % p.n_layers);
    const uint32_t bytes = p.chunks[c].bytes;
    mbar_arrive_expect_tx(bar_full + 8 * s, bytes);
    bulk_g2s(sb + L::kOffW + s * kStageBytes, p.wstream + (size_t)l * p.layer_bytes + p.chunks[c].off, bytes,
             bar_full + 8 * s);
    ++st.issued;
  }
}

// Wait until every warp has published the operand of GEMM `gemm`, issue its tcgen05.mma chain
// (accumulators at TMEM column 0), signal the accumulator barrier, then prefetch the next chunks.
template <int D>
__device__ __noinline__ void issue_gemm(const DecodeParams &p, const Ctl &ctl, IssueState &st, int gemm, uint32_t sb,
                                        uint32_t tmem) {
  using L = SmemLayout<D>;
  constexpr int S = L::kStages;
  const uint32_t bar_full = sb + L::kOffBar, bar_empty = bar_full + 8 * S;
  const uint32_t bar_op = bar_empty + 8 * S, bar_acc = bar_op + 8;
  wait_bar(ctl, bar_op, st.oph, false);
  st.oph ^= 1u;
  tc_fence_after();
  const uint32_t a_tile = (gemm == 3) ? (sb + L::kOffU) : (sb + L::kOffAop);
  const uint32_t a_sbo = (gemm == 3) ? (4u * D / 8u) * 128u : (D / 8u) * 128u;
  while (st.used < st.total) {
    const int c = static_cast<int>(st.used % p.n_chunks);
    const ChunkDesc ch = p.chunks[c];
    if (ch.gemm != gemm) break;
    issue_copies<D>(p, ctl, st, st.used + 1, sb);
    const int s = static_cast<int>(st.used % S);
    wait_bar(ctl, bar_full + 8 * s, static_cast<uint32_t>((st.used / S) & 1), false);
    tc_fence_after();
    const uint32_t b_tile = sb + L::kOffW + s * kStageBytes;
    const uint32_t b_sbo = (ch.kcols / 8u) * 128u;
    const uint32_t idesc = make_idesc_bf16(128, ch.nrows);
    for (int ks = 0; ks < ch.kcols / 16; ++ks) {
      const uint32_t kabs = ch.k0 + 16u * ks;
      const uint64_t ad = make_sdesc(a_tile + (kabs / 8u) * 128u, 128u, a_sbo);
      const uint64_t bd = make_sdesc(b_tile + ks * 256u, 128u, b_sbo);
      mma_bf16(tmem + ch.n0, ad, bd, idesc, kabs > 0 ? 1u : 0u);
    }
    mma_commit(bar_empty + 8 * s);
    ++st.used;
  }
  mma_commit(bar_acc);
  issue_copies<D>(p, ctl, st, st.used + S, sb);
}

// ------------------------------------------------------------------------------------------
// the kernel
// ------------------------------------------------------------------------------------------
template <int D>
__global__ void __launch_bounds__(kThreads, 1) aecct_decoder_kernel(const __grid_constant__ DecodeParams p) {
  using L = SmemLayout<D>;
  using LP = LayerParamLayout;
  constexpr int DH = D / kHeads;  // head width
  constexpr int XS = D / 4;       // x columns per thread
  constexpr int S = L::kStages;
  extern __shared__ __align__(1024) uint8_t smem[];
  const uint32_t sb = smem_u32(smem);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t crank = cluster_ctarank();
  const int cluster_id = blockIdx.x / p.C;

  const uint32_t bar_full = sb + L::kOffBar;
  const uint32_t bar_empty = bar_full + 8 * S;
  const uint32_t bar_op = bar_empty + 8 * S;
  const uint32_t bar_acc = bar_op + 8;
  const uint32_t bar_kvr = bar_acc + 8;
  const uint32_t bar_kvf = bar_kvr + 8;
  const uint32_t bar_zr = bar_kvf + 8;
  const uint32_t bar_zf = bar_zr + 8;
  const uint32_t bar_fin = bar_zf + 8;
  uint32_t *s_tmem = reinterpret_cast<uint32_t *>(smem + L::kOffMisc);
  volatile int *s_abort = reinterpret_cast<volatile int *>(smem + L::kOffMisc + 4);
  uint64_t *s_kvgen = reinterpret_cast<uint64_t *>(smem + L::kOffMisc + 8);  // [8] generic K/V bases per CTA
  uint64_t *s_zgen = reinterpret_cast<uint64_t *>(smem + L::kOffMisc + 72);   // [8] generic z bases per CTA

  if (tid == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(bar_full + 8 * s, 1);
      mbar_init(bar_empty + 8 * s, 1);
    }
    mbar_init(bar_op, kEpiWarps);
    mbar_init(bar_acc, 1);
    mbar_init(bar_kvr, p.C);
    mbar_init(bar_kvf, p.C);
    mbar_init(bar_zr, p.C);
    mbar_init(bar_zf, p.C);
    mbar_init(bar_fin, 1);
    *s_abort = 0;
    // generic base of the K/V and z areas of every CTA of the cluster: this CTA's own area through
    // its plain shared-memory window, the others through the distributed shared window
    for (int c = 0; c < p.C; ++c) {
      const bool own = c == static_cast<int>(crank);
      s_kvgen[c] = own ? reinterpret_cast<uint64_t>(smem + L::kOffU) : mapa_generic(smem + L::kOffU, c);
      s_zgen[c] = own ? reinterpret_cast<uint64_t>(smem + L::kOffZ) : mapa_generic(smem + L::kOffZ, c);
    }
    fence_mbar_init_cluster();
  }
  __syncwarp();  // warp 0 reconverges before its warp-collective TMEM allocation
  if (warp == 0) {
    tmem_alloc(smem_u32(s_tmem), L::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  cluster_sync_all();
  tc_fence_after();
  const uint32_t tmem = *s_tmem;
  const Ctl ctl{s_abort, p.err, p.wait_limit};

  IssueState ist{0, 0, 0, 0};
  if (tid == 0) {
    const int64_t my_groups = (p.n_groups - cluster_id + p.n_clusters - 1) / p.n_clusters;
    ist.total = my_groups * p.n_layers * p.n_chunks;
    issue_copies<D>(p, ctl, ist, S, sb);
  }
  __syncwarp();
  {
    // ------------------------------------------------------------ CUDA-core warps
    const int qd = warp & 3, sl = warp >> 2;
    const int r = 32 * qd + lane;
    const uint32_t tl = tmem + (static_cast<uint32_t>(32 * qd) << 16);
    const uint32_t aop = sb + L::kOffAop;
    const uint32_t uqt = sb + L::kOffU;
    const uint32_t kvl = sb + L::kOffU;
    RowRed red{reinterpret_cast<float *>(smem + L::kOffRed), 0};
    float *zbuf = reinterpret_cast<float *>(smem + L::kOffZ);
    uint8_t *obits = smem + L::kOffObits;
    const uint32_t qbar = 1 + qd;  // named barrier of the 4 warps sharing a lane quadrant
    const int T = p.T, n = p.n, m = p.m, de = D - p.d_spe;
    const int W4 = 4 * D;
    const float inv_d = 1.0f / static_cast<float>(D);
    uint32_t acc_ph = 0, kvr_ph = 0, kvf_ph = 0, zr_ph = 0;
    int64_t z_uses = 0;

    // reduce one value per row over the 4 slices: max or pairwise sum ((s0+s1)+(s2+s3))
    auto row_max = [&](float v) -> float {
      *red.slot(sl, r) = v;
      named_bar_sync(qbar, 128);
      const float a = fmaxf(fmaxf(*red.slot(0, r), *red.slot(1, r)), fmaxf(*red.slot(2, r), *red.slot(3, r)));
      red.sel ^= 1;
      return a;
    };
    auto row_sum = [&](float v) -> float {
      *red.slot(sl, r) = v;
      named_bar_sync(qbar, 128);
      const float a = __fadd_rn(__fadd_rn(*red.slot(0, r), *red.slot(1, r)), __fadd_rn(*red.slot(2, r), *red.slot(3, r)));
      red.sel ^= 1;
      return a;
    };
    // publish this warp's part of the operand of `gemm`; thread 0 then issues the GEMM
    auto signal_op = [&](int gemm) {
      tc_fence_before();  // this thread's TMEM reads are ordered before the MMA the arrive releases
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(bar_op);
      if (tid == 0) issue_gemm<D>(p, ctl, ist, gemm, sb, tmem);
      __syncwarp();  // warp 0 waits for its issuing lane before any warp-collective instruction
    };
    auto cluster_arrive = [&](uint32_t bar) {
      // all 512 CUDA-core threads of this CTA are past their accesses: tell every CTA
      named_bar_sync(5, kEpiThreads);
      if (tid == 0) {
        fence_acq_rel_cluster();
        for (int c = 0; c < p.C; ++c) mbar_arrive_cluster(mapa_cluster(bar, c));
      }
      __syncwarp();
    };
    auto wait_acc = [&]() {
      wait_bar(ctl, bar_acc, acc_ph, false);
      acc_ph ^= 1u;
      tc_fence_after();
    };

    for (int64_t gi = cluster_id; gi < p.n_groups; gi += p.n_clusters) {
      if (named_bar_or(5, kEpiThreads, *s_abort != 0)) break;
      const int rho = static_cast<int>(crank) * kRows + r;
      const int g = rho / T;
      const int t = __ldg(p.perm + (rho - g * T));  // token held by this row (rows are ordered by attention work)
      const int64_t b = gi * p.G + g;
      const bool row_cw = g < p.G;
      const bool valid = row_cw && b < p.B;
      const bool cap = valid && b < p.cap_B;
      const float *yrow = p.y + (valid ? b : 0) * n;

      float x[XS];
      float alpha_in;
      // ---------------- S1/S2: tokens, embedding, SPE (Sec. 3, Sec. 4.3)
      {
        float h = 0.0f;
        if (valid) {
          if (t < n) {
            h = fabsf(__ldg(yrow + t));
          } else {
            const int i = t - n;
            uint32_t par = 0;
            for (uint32_t e = __ldg(p.hrow_off + i); e < __ldg(p.hrow_off + i + 1); ++e)
              par ^= (__ldg(yrow + __ldg(p.hrow_idx + e)) < 0.0f) ? 1u : 0u;
            h = __fsub_rn(1.0f, __fmul_rn(2.0f, static_cast<float>(par)));
            if (cap && sl == 0 && p.cap_syn) p.cap_syn[b * m + i] = static_cast<uint8_t>(par);
          }
        }
#pragma unroll
        for (int j = 0; j < XS; ++j) {
          const int c = sl * XS + j;
          float v = 0.0f;
          if (valid) v = (c < de) ? __fmul_rn(h, __ldg(p.emb + t * de + c)) : __ldg(p.spe + t * p.d_spe + (c - de));
          x[j] = v;
        }
      }
      // Quant(x) -> QKV operand (Sec. 4.1 eq. Quant)
      auto quant_x_to_aop = [&]() -> float {
        float a = 0.0f;
#pragma unroll
        for (int j = 0; j < XS; ++j) a = fmaxf(a, fabsf(x[j]));
        a = row_max(a);
        a = (a > p.alpha_floor) ? a : p.alpha_floor;
        alpha_in = a;
        const float rr = __fdiv_rn(127.0f, a);
        float qv[XS];
#pragma unroll
        for (int j = 0; j < XS; ++j) qv[j] = q_code(x[j], rr);
        store_codes<XS>(aop, r, sl * XS, D, qv);
        return rr;
      };
      auto capture_q = [&](int layer, int gemm, const float *qv, int c0, int len, float alpha) {
        const int64_t row = ((b * p.n_layers + layer) * 4 + gemm) * T + t;
        if (p.cap_q)
          for (int j = 0; j < len; ++j) p.cap_q[row * W4 + c0 + j] = static_cast<int8_t>(qv[j]);
        if (p.cap_alpha && sl == 0) p.cap_alpha[row] = alpha;
      };
      auto capture_acc = [&](int layer, int gemm, const float *av, int c0, int len) {
        const int64_t row = ((b * p.n_layers + layer) * 4 + gemm) * T + t;
        if (p.cap_acc)
          for (int j = 0; j < len; ++j) p.cap_acc[row * W4 + c0 + j] = static_cast<int32_t>(av[j]);
      };

      {
        const float rr = quant_x_to_aop();
        if (cap) {
          float qv[XS];
#pragma unroll
          for (int j = 0; j < XS; ++j) qv[j] = q_code(x[j], rr);
          capture_q(0, 0, qv, sl * XS, XS, alpha_in);
        }
      }
      signal_op(0);

      for (int l = 0; l < p.n_layers; ++l) {
        const float *lp = p.lparams + (size_t)l * LP::stride(D);
        const float *sw = lp + LP::sw(D);
        // ---------------- S4 epilogue: K, V to shared memory
        wait_acc();
        // park the residual row in TMEM columns [3D, 4D) (unused by the QKV and O accumulators)
        // so that attention runs with the registers it needs
        tmem_st<XS>(tl + 3 * D + sl * XS, x);
        tmem_wait_st();
        const float fq = __fdiv_rn(__fmul_rn(__ldg(sw + 0), alpha_in), 127.0f);
        const float fk = __fdiv_rn(__fmul_rn(__ldg(sw + 1), alpha_in), 127.0f);
        const float fv = __fdiv_rn(__fmul_rn(__ldg(sw + 2), alpha_in), 127.0f);
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
          const int e = sl + 4 * hh;
          float ka[DH], va[DH], bk[DH], bv[DH];
          tmem_ld<DH>(tl + D + e * DH, ka);
          tmem_ld<DH>(tl + 2 * D + e * DH, va);
          tmem_wait_ld();
          ldg_vec<DH>(lp + LP::bqkv(D) + D + e * DH, bk);
          ldg_vec<DH>(lp + LP::bqkv(D) + 2 * D + e * DH, bv);
          if (cap) {
            capture_acc(l, 0, ka, D + e * DH, DH);
            capture_acc(l, 0, va, 2 * D + e * DH, DH);
          }
          const uint32_t dst = kvl + r * L::kKvStride + e * (8 * DH);
#pragma unroll
          for (int i = 0; i < DH; i += 4) {
            st_shared_f4(dst + 4 * i, __fadd_rn(__fmul_rn(ka[i], fk), bk[i]), __fadd_rn(__fmul_rn(ka[i + 1], fk), bk[i + 1]),
                         __fadd_rn(__fmul_rn(ka[i + 2], fk), bk[i + 2]), __fadd_rn(__fmul_rn(ka[i + 3], fk), bk[i + 3]));
            st_shared_f4(dst + 4 * (DH + i), __fadd_rn(__fmul_rn(va[i], fv), bv[i]),
                         __fadd_rn(__fmul_rn(va[i + 1], fv), bv[i + 1]), __fadd_rn(__fmul_rn(va[i + 2], fv), bv[i + 2]),
                         __fadd_rn(__fmul_rn(va[i + 3], fv), bv[i + 3]));
          }
        }
        cluster_arrive(bar_kvr);
        wait_bar(ctl, bar_kvr, kvr_ph, true);
        kvr_ph ^= 1u;

        // ---------------- S5: HPSA (Sec. 4.2)
        float A[2][DH];
        float amax = 0.0f;
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
          const int e = sl + 4 * hh;
          float qa[DH], bq[DH];
          tmem_ld<DH>(tl + e * DH, qa);
          tmem_wait_ld();
          if (cap) capture_acc(l, 0, qa, e * DH, DH);
          ldg_vec<DH>(lp + LP::bqkv(D) + e * DH, bq);
          float q[DH];
#pragma unroll
          for (int i = 0; i < DH; ++i) q[i] = __fadd_rn(__fmul_rn(qa[i], fq), bq[i]);
#pragma unroll
          for (int i = 0; i < DH; ++i) A[hh][i] = 0.0f;
          if (row_cw) {
            const int mk = (e < p.h_first) ? 0 : 1;
            constexpr int U = (DH >= 16) ? 2 : 4;
            hpsa_head<DH, U, L::kKvStride>(q, __ldg(p.mask_info[mk] + t), p.mask_list[mk], s_kvgen, g * T,
                                           e * (8 * DH), p.att_scale, A[hh]);
          }
          __syncwarp();  // lanes leave their key loops at different times; reconverge before tcgen05.ld
#pragma unroll
          for (int i = 0; i < DH; ++i) amax = fmaxf(amax, fabsf(A[hh][i]));
        }
        // Quant(A) -> O operand
        {
          float a = row_max(amax);
          a = (a > p.alpha_floor) ? a : p.alpha_floor;
          alpha_in = a;
          const float rr = __fdiv_rn(127.0f, a);
#pragma unroll
          for (int hh = 0; hh < 2; ++hh) {
            const int e = sl + 4 * hh;
            float qv[DH];
#pragma unroll
            for (int i = 0; i < DH; ++i) qv[i] = q_code(A[hh][i], rr);
            store_codes<DH>(aop, r, e * DH, D, qv);
            if (cap) capture_q(l, 1, qv, e * DH, DH, alpha_in);
          }
        }
        signal_op(1);
        cluster_arrive(bar_kvf);  // this CTA no longer reads any K/V of this block

        // ---------------- S6: O projection + residual + LayerNorm (Sec. 5, Post-LN)
        wait_acc();
        {
          const float fo = __fdiv_rn(__fmul_rn(__ldg(sw + 3), alpha_in), 127.0f);
          float ac[XS], bb[XS], gg[XS], be[XS];
          tmem_ld<XS>(tl + sl * XS, ac);
          tmem_ld<XS>(tl + 3 * D + sl * XS, x);
          tmem_wait_ld();
          if (cap) capture_acc(l, 1, ac, sl * XS, XS);
          ldg_vec<XS>(lp + LP::bo(D) + sl * XS, bb);
          float v[XS];
#pragma unroll
          for (int j = 0; j < XS; ++j) v[j] = __fadd_rn(x[j], __fadd_rn(__fmul_rn(ac[j], fo), bb[j]));
          const float mu = __fmul_rn(row_sum(psum<XS>(v)), inv_d);
#pragma unroll
          for (int j = 0; j < XS; ++j) {
            v[j] = __fsub_rn(v[j], mu);
            ac[j] = __fmul_rn(v[j], v[j]);
          }
          const float var = __fmul_rn(row_sum(psum<XS>(ac)), inv_d);
          const float rstd = __fdiv_rn(1.0f, __fsqrt_rn(__fadd_rn(var, p.ln_eps)));
          ldg_vec<XS>(lp + LP::ln1g(D) + sl * XS, gg);
          ldg_vec<XS>(lp + LP::ln1b(D) + sl * XS, be);
#pragma unroll
          for (int j = 0; j < XS; ++j) x[j] = __fadd_rn(__fmul_rn(__fmul_rn(v[j], rstd), gg[j]), be[j]);
        }
        {
          const float rr = quant_x_to_aop();
          if (cap) {
            float qv[XS];
#pragma unroll
            for (int j = 0; j < XS; ++j) qv[j] = q_code(x[j], rr);
            capture_q(l, 2, qv, sl * XS, XS, alpha_in);
          }
        }
        signal_op(2);

        // ---------------- S7: FFN1 + ReLU (Sec. 4 item 4), Quant(u) -> FFN2 operand
        wait_acc();
        {
          const float f1 = __fdiv_rn(__fmul_rn(__ldg(sw + 4), alpha_in), 127.0f);
          constexpr int NCH = D / 32;  // 32-column chunks of this thread's D hidden columns
          float umax = 0.0f;
#pragma unroll 1
          for (int ch = 0; ch < NCH; ++ch) {
            const int c0 = sl * D + 32 * ch;
            float ac[32], bb[32];
            tmem_ld<32>(tl + c0, ac);
            tmem_wait_ld();
            if (cap) capture_acc(l, 2, ac, c0, 32);
            ldg_vec<32>(lp + LP::b1(D) + c0, bb);
#pragma unroll
            for (int j = 0; j < 32; ++j) {
              float u = __fadd_rn(__fmul_rn(ac[j], f1), bb[j]);
              u = u > 0.0f ? u : 0.0f;
              umax = fmaxf(umax, u);
            }
          }
          float a = row_max(umax);
          a = (a > p.alpha_floor) ? a : p.alpha_floor;
          alpha_in = a;
          const float rr = __fdiv_rn(127.0f, a);
          // peers have finished reading this CTA's K/V: the shared region may now take u codes
          wait_bar(ctl, bar_kvf, kvf_ph, true);
          kvf_ph ^= 1u;
#pragma unroll 1
          for (int ch = 0; ch < NCH; ++ch) {
            const int c0 = sl * D + 32 * ch;
            float ac[32], bb[32];
            tmem_ld<32>(tl + c0, ac);
            tmem_wait_ld();
            ldg_vec<32>(lp + LP::b1(D) + c0, bb);
            float qv[32];
#pragma unroll
            for (int j = 0; j < 32; ++j) {
              float u = __fadd_rn(__fmul_rn(ac[j], f1), bb[j]);
              u = u > 0.0f ? u : 0.0f;
              qv[j] = q_code(u, rr);
            }
            store_codes<32>(uqt, r, c0, 4 * D, qv);
            if (cap) capture_q(l, 3, qv, c0, 32, alpha_in);
          }
        }
        signal_op(3);

        // ---------------- S8: FFN2 + residual + LayerNorm
        wait_acc();
        {
          const float f2 = __fdiv_rn(__fmul_rn(__ldg(sw + 5), alpha_in), 127.0f);
          float ac[XS], bb[XS], gg[XS], be[XS];
          tmem_ld<XS>(tl + sl * XS, ac);
          tmem_wait_ld();
          if (cap) capture_acc(l, 3, ac, sl * XS, XS);
          ldg_vec<XS>(lp + LP::b2(D) + sl * XS, bb);
          float v[XS];
#pragma unroll
          for (int j = 0; j < XS; ++j) v[j] = __fadd_rn(x[j], __fadd_rn(__fmul_rn(ac[j], f2), bb[j]));
          const float mu = __fmul_rn(row_sum(psum<XS>(v)), inv_d);
#pragma unroll
          for (int j = 0; j < XS; ++j) {
            v[j] = __fsub_rn(v[j], mu);
            ac[j] = __fmul_rn(v[j], v[j]);
          }
          const float var = __fmul_rn(row_sum(psum<XS>(ac)), inv_d);
          const float rstd = __fdiv_rn(1.0f, __fsqrt_rn(__fadd_rn(var, p.ln_eps)));
          ldg_vec<XS>(lp + LP::ln2g(D) + sl * XS, gg);
          ldg_vec<XS>(lp + LP::ln2b(D) + sl * XS, be);
#pragma unroll
          for (int j = 0; j < XS; ++j) x[j] = __fadd_rn(__fmul_rn(__fmul_rn(v[j], rstd), gg[j]), be[j]);
        }
        if (l + 1 < p.n_layers) {
          const float rr = quant_x_to_aop();
          if (cap) {
            float qv[XS];
#pragma unroll
            for (int j = 0; j < XS; ++j) qv[j] = q_code(x[j], rr);
            capture_q(l + 1, 0, qv, sl * XS, XS, alpha_in);
          }
          signal_op(0);
        }
      }

      // ---------------- S9: output head (Sec. 3): z_t = x_t . w_{d->1} + b, eps = W_o^T z + b_o
      {
        float wv[XS];
        ldg_vec<XS>(p.w_d1 + sl * XS, wv);
#pragma unroll
        for (int j = 0; j < XS; ++j) wv[j] = __fmul_rn(x[j], wv[j]);
        const float z = __fadd_rn(row_sum(psum<XS>(wv)), p.b_d1);
        if (z_uses > 0) wait_bar(ctl, bar_zf, static_cast<uint32_t>((z_uses - 1) & 1), true);
        ++z_uses;
        if (sl == 0) zbuf[r] = z;
      }
      cluster_arrive(bar_zr);
      wait_bar(ctl, bar_zr, zr_ph, true);
      zr_ph ^= 1u;
      // ---------------- S10: decisions x_hat = y * eps, decoded-word syndrome
      {
        const int n_local = (p.G - static_cast<int>(crank) + p.C - 1) / p.C;  // groups g = crank + C*i
        const int items = n_local * n;
        for (int it = tid; it < items; it += kEpiThreads) {
          const int li = it / n, j = it - li * n;
          const int gg = static_cast<int>(crank) + li * p.C;
          const int64_t bb = gi * p.G + gg;
          if (bb >= p.B) continue;
          float acc = 0.0f;
          const int rb0 = gg * T;
          for (int tt = 0; tt < T; ++tt) {
            const int ru = rb0 + __ldg(p.pos + tt);
            const float zt = *reinterpret_cast<const float *>(s_zgen[ru >> 7] + static_cast<uint32_t>(ru & 127) * 4u);
            acc = __fmaf_rn(__ldg(p.w_out + tt * n + j), zt, acc);
          }
          const float eps = __fadd_rn(acc, __ldg(p.b_out + j));
          const uint8_t bit = (__fmul_rn(__ldg(p.y + bb * n + j), eps) < 0.0f) ? 1 : 0;
          p.bits[bb * n + j] = bit;
          if (p.logits) p.logits[bb * n + j] = eps;
          obits[li * n + j] = bit;
        }
        named_bar_sync(5, kEpiThreads);
        if (p.syn) {
          const int sitems = n_local * m;
          for (int it = tid; it < sitems; it += kEpiThreads) {
            const int li = it / m, i = it - li * m;
            const int gg = static_cast<int>(crank) + li * p.C;
            const int64_t bb = gi * p.G + gg;
            if (bb >= p.B) continue;
            uint32_t par = 0;
            for (uint32_t e = __ldg(p.hrow_off + i); e < __ldg(p.hrow_off + i + 1); ++e)
              par ^= obits[li * n + __ldg(p.hrow_idx + e)];
            p.syn[bb * m + i] = static_cast<uint8_t>(par);
          }
        }
        cluster_arrive(bar_zf);  // this CTA no longer reads any z of this group; obits free
      }
    }
  }

  // ------------------------------------------------------------ teardown
  if (tid == 0) {
    // every MMA and every weight copy this CTA started must have landed before TMEM and the
    // shared memory go away
    mma_commit(bar_fin);
    wait_bar_drain(ctl, bar_fin, 0);
    for (int64_t i = ist.issued - S; i < ist.issued; ++i)
      if (i >= 0) wait_bar_drain(ctl, bar_full + 8 * static_cast<int>(i % S), static_cast<uint32_t>((i / S) & 1));
  }
  tc_fence_before();
  __syncwarp();
  cluster_sync_all();
  if (warp == 0) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, L::kTmemCols);
  }
}

template <int D>
cudaError_t prepare_decode_kernel(int cluster_ctas, int *max_active_clusters) {
  using L = SmemLayout<D>;
  cudaError_t e = cudaFuncSetAttribute(aecct_decoder_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(L::kTotal));
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = cluster_ctas;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.gridDim = dim3(cluster_ctas, 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = L::kTotal;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaOccupancyMaxActiveClusters(max_active_clusters, aecct_decoder_kernel<D>, &cfg);
}

template <int D>
cudaError_t launch_decode(const DecodeParams &p, cudaStream_t stream) {
  using L = SmemLayout<D>;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = p.C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.gridDim = dim3(p.n_clusters * p.C, 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = L::kTotal;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, aecct_decoder_kernel<D>, p);
}

template cudaError_t launch_decode<32>(const DecodeParams &, cudaStream_t);
template cudaError_t launch_decode<64>(const DecodeParams &, cudaStream_t);
template cudaError_t launch_decode<128>(const DecodeParams &, cudaStream_t);
template cudaError_t prepare_decode_kernel<32>(int, int *);
template cudaError_t prepare_decode_kernel<64>(int, int *);
template cudaError_t prepare_decode_kernel<128>(int, int *);

}  // namespace aecct
