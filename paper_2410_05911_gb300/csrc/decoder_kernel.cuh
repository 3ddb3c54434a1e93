// decoder_kernel.cuh -- the fused AECCT forward pass for sm_103a (kernel template; its
// instantiations live in decoder_kernel.cu (ReLU, AAP linears), decoder_kernel_gelu.cu (GELU),
// decoder_kernel_fp.cu and decoder_kernel_fp_gelu.cu (full-precision bf16 linears), translation
// units that compile in parallel).
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
//          -> HPSA (warp tasks over shared key lists, or per-row neighbour lists with
//          distributed-shared-memory reads of peer CTAs) -> Quant(A) -> MMA O
//          -> dequant + residual + LayerNorm -> Quant -> MMA FFN1 -> dequant + ReLU/GELU ->
//          Quant -> MMA FFN2 -> dequant + residual + LayerNorm
//   S9/S10 (Sec. 3)        output head, hard decisions, syndrome of the decoded word
//
// Warp roles (512 threads): warps 0-15 do all CUDA-core work; thread (warp w, lane i) owns
// token row 32*(w%4) + i (the TMEM lane quadrant its warp may read) and column slice w/4.
// Between its CUDA-core steps, warp 0 also streams the block weights from global memory into
// a ring of shared-memory stages with the bulk-copy (TMA) engine and issues the tensor-core
// MMAs, in a compile-time schedule (WeightSchedule).
//
// Every floating-point step uses one fixed order of IEEE fp32 operations (explicit _rn
// intrinsics, pairwise feature sums, two-pass base-2 softmax with a Taylor-series exp2), so
// the results are bit-identical to any implementation that follows the same order.
#pragma once
#include <cuda_runtime.h>

#include <type_traits>

#include "aecct_internal.h"
#include "sm103_ptx.cuh"

namespace aecct {

// fp32(ln(2)^k / k!), k = 0..7: Taylor coefficients of 2^f = e^(f ln 2)
__device__ __forceinline__ float exp2_series(float x) {
  if (!(x >= -125.0f)) return 0.0f;
  // n = rint(x) through the rounding add (x is in [-125, 0] here); the integer n also sits in the
  // low bits of t, which gives the exponent shift without a conversion
  const float t = __fadd_rn(x, 12582912.0f);
  const float n = __fsub_rn(t, 12582912.0f);
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
  return __int_as_float(__float_as_int(p) + ((__float_as_int(t) - 0x4B400000) << 23));
}

// GELU(x) = x Phi(x) = 0.5 x (1 + erf(x / sqrt 2)), the feed-forward activation option.  erf is
// the rational approximation of Abramowitz & Stegun, Handbook of Mathematical Functions, formula
// 7.1.26 (|error| <= 1.5e-7 for x >= 0; odd symmetry for x < 0), with its exponential through
// exp2_series:  z = x fp32(1/sqrt 2), t = 1 / (1 + p|z|),
// erf|z| = 1 - t (a1 + t (a2 + t (a3 + t (a4 + t a5)))) 2^(z^2 fp32(-log2 e)).
__device__ __forceinline__ float gelu_as(float x) {
  const float z = __fmul_rn(x, 0.70710678118654752f);
  const float az = fabsf(z);
  const float t = __fdiv_rn(1.0f, __fmaf_rn(0.3275911f, az, 1.0f));
  float q = 1.061405429f;
  q = __fmaf_rn(q, t, -1.453152027f);
  q = __fmaf_rn(q, t, 1.421413741f);
  q = __fmaf_rn(q, t, -0.284496736f);
  q = __fmaf_rn(q, t, 0.254829592f);
  q = __fmul_rn(q, t);
  const float e = exp2_series(__fmul_rn(__fmul_rn(az, az), -1.44269504088896341f));
  const float er = __fsub_rn(1.0f, __fmul_rn(q, e));
  return __fmul_rn(__fmul_rn(0.5f, x), __fadd_rn(1.0f, z < 0.0f ? -er : er));
}

// ---- paired fp32 arithmetic (sm_100 f32x2: each lane is one IEEE round-to-nearest operation,
// bit-identical to the scalar _rn operation on that lane).  The code generator contracts a paired
// multiply whose only use is a paired add into one fused multiply-add, even with --fmad=false
// and an explicit .rn modifier, so pairs are used only where no contraction can occur: fused
// multiply-adds that the canonical order asks for, adds of values that are not products, and
// products that feed no add.  Every multiply-then-add of the canonical order uses the scalar
// __fmul_rn / __fadd_rn intrinsics, which are never contracted.
__device__ __forceinline__ uint64_t pack2(float2 a) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(a.x), "f"(a.y));
  return r;
}
__device__ __forceinline__ float2 unpack2(uint64_t r) {
  float2 a;
  asm("mov.b64 {%0, %1}, %2;" : "=f"(a.x), "=f"(a.y) : "l"(r));
  return a;
}
__device__ __forceinline__ float2 mul2(float2 a, float2 b) {
  uint64_t d;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(pack2(a)), "l"(pack2(b)));
  return unpack2(d);
}
__device__ __forceinline__ float2 add2(float2 a, float2 b) {
  uint64_t d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(pack2(a)), "l"(pack2(b)));
  return unpack2(d);
}
__device__ __forceinline__ float2 fma2(float2 a, float2 b, float2 c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(pack2(a)), "l"(pack2(b)), "l"(pack2(c)));
  return unpack2(d);
}

// two independent evaluations of exp2_series (same steps on each lane); inputs below -125 give 0
__device__ __forceinline__ float2 exp2_series2(float2 x) {
  const float2 t = add2(x, make_float2(12582912.0f, 12582912.0f));  // rounding adds, as in exp2_series
  const float2 nn = add2(t, make_float2(-12582912.0f, -12582912.0f));
  const float2 f = add2(x, make_float2(-nn.x, -nn.y));
  float2 p = make_float2(__uint_as_float(0x377fe5feu), __uint_as_float(0x377fe5feu));
  p = fma2(p, f, make_float2(__uint_as_float(0x39218489u), __uint_as_float(0x39218489u)));
  p = fma2(p, f, make_float2(__uint_as_float(0x3aaec3ffu), __uint_as_float(0x3aaec3ffu)));
  p = fma2(p, f, make_float2(__uint_as_float(0x3c1d955bu), __uint_as_float(0x3c1d955bu)));
  p = fma2(p, f, make_float2(__uint_as_float(0x3d635847u), __uint_as_float(0x3d635847u)));
  p = fma2(p, f, make_float2(__uint_as_float(0x3e75fdf0u), __uint_as_float(0x3e75fdf0u)));
  p = fma2(p, f, make_float2(__uint_as_float(0x3f317218u), __uint_as_float(0x3f317218u)));
  p = fma2(p, f, make_float2(1.0f, 1.0f));
  const float r0 = (x.x >= -125.0f) ? __int_as_float(__float_as_int(p.x) + ((__float_as_int(t.x) - 0x4B400000) << 23)) : 0.0f;
  const float r1 = (x.y >= -125.0f) ? __int_as_float(__float_as_int(p.y) + ((__float_as_int(t.y) - 0x4B400000) << 23)) : 0.0f;
  return make_float2(r0, r1);
}

// out[j] = acc[j] * f + b[j]  (eq. AAPLinear dequantisation, f = gamma*delta*alpha/Q_b): a
// separately rounded product, then the bias add; the adds of two outputs run as one paired add
// (the products stay scalar multiplies, so nothing is fused)
template <int N>
__device__ __forceinline__ void dequant(const float *acc, float f, const float *b, float *out) {
  static_assert(N % 2 == 0, "pairs");
#pragma unroll
  for (int j = 0; j < N; j += 2) {
    const float2 o = add2(make_float2(__fmul_rn(acc[j], f), __fmul_rn(acc[j + 1], f)), make_float2(b[j], b[j + 1]));
    out[j] = o.x, out[j + 1] = o.y;
  }
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

// Bounded mbarrier wait (wait_bar).  Returns false (and raises the CTA abort flag plus the
// device error word) when the phase does not complete within `limit` SM cycles; once the abort
// flag is up every later wait returns false at once so the kernel drains without blocking.
// The polling loop is out of line; the first test is inline (a call saves registers to local
// memory, which misses the small L1 left beside the shared-memory carve-out).
static __device__ __noinline__ bool wait_bar_slow(const Ctl c, uint32_t bar, uint32_t parity, bool cluster_scope) {
  const long long t0 = clock64();
  while (true) {
    if (cluster_scope ? mbar_try_wait_acq_cluster(bar, parity) : mbar_try_wait(bar, parity)) return true;
    if (*c.abort) return false;
    if (clock64() - t0 > c.limit) {
      *c.abort = 1;
      atomicOr(c.err, 1);
      return false;
    }
  }
}
__device__ __forceinline__ bool wait_bar(const Ctl c, uint32_t bar, uint32_t parity, bool cluster_scope) {
  if (*c.abort) return false;
  if (cluster_scope ? mbar_try_wait_acq_cluster(bar, parity) : mbar_try_wait(bar, parity)) return true;
  return wait_bar_slow(c, bar, parity, cluster_scope);
}
// The same wait for a whole converged warp: lane 0 polls, the result goes to every lane.
__device__ __forceinline__ bool wait_bar_warp(const Ctl c, uint32_t bar, uint32_t parity, bool cluster_scope) {
  bool ok = true;
  if ((threadIdx.x & 31) == 0) ok = wait_bar(c, bar, parity, cluster_scope);
  return __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
}
// Teardown wait: ignores the abort flag (used to drain copies / MMAs in flight).  Its bound is
// fixed (about a second) and independent of the caller's wait limit: the copies and MMAs it waits
// for were all issued on the live path (the issuer stops issuing once a wait gave up), so they
// finish in microseconds, and a short caller limit must not let the kernel exit while a copy can
// still land in its shared memory.
constexpr long long kDrainLimitCycles = 1LL << 31;
static __device__ __noinline__ bool wait_bar_drain(const Ctl c, uint32_t bar, uint32_t parity) {
  const long long t0 = clock64();
  while (!mbar_try_wait(bar, parity)) {
    if (clock64() - t0 > kDrainLimitCycles) {
      atomicOr(c.err, 1);
      return false;
    }
  }
  return true;
}

// ------------------------------------------------------------------------------------------
// small helpers for the CUDA-core warps
// ------------------------------------------------------------------------------------------
// Round to the nearest integer, ties to even, for |x| < 2^22, on the FP32 add pipe: x + 1.5 * 2^23
// lies in [2^23, 2^24), where the spacing of fp32 values is 1, so the round-to-nearest-even add
// rounds x exactly as rintf does, and subtracting 1.5 * 2^23 back is exact.  (rintf runs on the
// quarter-rate conversion pipe.)
constexpr float kRoundMagic = 12582912.0f;  // 1.5 * 2^23
__device__ __forceinline__ float round_even(float x) { return __fsub_rn(__fadd_rn(x, kRoundMagic), kRoundMagic); }

// Code of v under r = 127/alpha' (eq. Quant).  |v| <= alpha' gives |v * r| <= 127 (1 + 2^-24)
// before rounding, so the clip of RoundClip can never act and is left out.  The product stays a
// separately rounded scalar multiply (a paired multiply feeding the rounding add would be fused).
__device__ __forceinline__ float q_code(float v, float r) { return round_even(__fmul_rn(v, r)); }
// the codes of N values (N even): the products stay separately rounded scalar multiplies, and
// the two rounding adds of a pair of codes run as paired adds (adds of values that are not paired
// products, so nothing is fused); the same codes as q_code
template <int N>
__device__ __forceinline__ void codes(const float *v, float r, float *q) {
  static_assert(N % 2 == 0, "pairs");
#pragma unroll
  for (int j = 0; j < N; j += 2) {
    const float2 t = add2(make_float2(__fmul_rn(v[j], r), __fmul_rn(v[j + 1], r)),
                          make_float2(kRoundMagic, kRoundMagic));
    const float2 c = add2(t, make_float2(-kRoundMagic, -kRoundMagic));
    q[j] = c.x, q[j + 1] = c.y;
  }
}
__device__ __forceinline__ uint32_t pack_bf16x2(float a, float b) {
  // a, b are integers in [-127, 127]: their fp32 encodings have 16 zero low bits, so the bf16
  // encodings are the high halves (one byte permute instead of two conversions)
  return __byte_perm(__float_as_uint(a), __float_as_uint(b), 0x7632);
}
__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
  asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(a), "r"(b), "r"(c), "r"(d) : "memory");
}
__device__ __forceinline__ void st_shared_v2(uint32_t addr, uint32_t a, uint32_t b) {
  asm volatile("st.shared.v2.b32 [%0], {%1, %2};" ::"r"(addr), "r"(a), "r"(b) : "memory");
}
__device__ __forceinline__ float4 ld_shared_f4(uint32_t addr) {
  float4 v;
  asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];" : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w) : "r"(addr) : "memory");
  return v;
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

// write LEN consecutive fp32 values of row r, rounded to bf16 (round to nearest even), into a
// K-major operand tile (full-precision linears)
__device__ __forceinline__ uint32_t pack_bf16x2_rn(float a, float b) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(a, b);  // a in the low half
  return *reinterpret_cast<const uint32_t *>(&v);
}
template <int LEN>
__device__ __forceinline__ void store_bf16(uint32_t tile, int r, int c0, int kdim, const float *v) {
  if constexpr (LEN == 4) {
    st_shared_v2(tile + core_off(r, c0, kdim), pack_bf16x2_rn(v[0], v[1]), pack_bf16x2_rn(v[2], v[3]));
  } else {
    static_assert(LEN % 8 == 0, "bf16 run");
#pragma unroll
    for (int j = 0; j < LEN; j += 8)
      st_shared_v4(tile + core_off(r, c0 + j, kdim), pack_bf16x2_rn(v[j], v[j + 1]),
                   pack_bf16x2_rn(v[j + 2], v[j + 3]), pack_bf16x2_rn(v[j + 4], v[j + 5]),
                   pack_bf16x2_rn(v[j + 6], v[j + 7]));
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
// Every lane has its own list; the warp walks 8-key blocks up to the longest list of its lanes
// (a lane past its own count computes on a valid dummy row and folds nothing in).  The scores of
// the first kRowCache keys go to this thread's TMEM columns in pass 1 and come back in pass 2, in
// place of a second load of K and a second dot product (the same fp32 values).
// K (then V) row of one head, as float4s: in this CTA's shared memory (one-CTA cluster; plain
// loads the compiler schedules) or in the CTA of the cluster that holds the row (32-bit
// shared::cluster address)
template <bool CLUSTER>
struct KeyRow;
template <>
struct KeyRow<false> {
  const float4 *p;
  __device__ __forceinline__ float4 operator[](int i) const { return p[i]; }
};
template <>
struct KeyRow<true> {
  uint32_t a;
  __device__ __forceinline__ float4 operator[](int i) const { return ld_cluster_f32x4(a + 16u * i); }
};

template <int DH, int U, uint32_t STRIDE, bool CLUSTER>
__device__ __forceinline__ void hpsa_head(const float *q, uint32_t info, bool active, const uint4 *__restrict__ lists,
                                          const uint8_t *kvlocal, const uint32_t *kvbase, int rowbase,
                                          uint32_t hoff, float scale, uint32_t tcache, float *A) {
  static_assert(8 % U == 0, "keys per index block");
  const uint4 *lst = lists + (info >> 11);
  const int cnt = active ? static_cast<int>(info & 2047u) : 0;
  const int nmax = __reduce_max_sync(0xffffffffu, cnt);
  // K (then V) of key row `off` of this head, from the CTA that holds it
  auto keyptr = [&](int off) -> KeyRow<CLUSTER> {
    const int ru = rowbase + off;
    if constexpr (CLUSTER)
      return KeyRow<true>{kvbase[ru >> 7] + static_cast<uint32_t>(ru & 127) * STRIDE + hoff};
    else
      return KeyRow<false>{reinterpret_cast<const float4 *>(kvlocal + static_cast<uint32_t>(ru) * STRIDE + hoff)};
  };
  // q . k in the canonical order: even-feature and odd-feature FMA chains (the two lanes of
  // paired FMAs over adjacent features), then their sum
  auto dotk = [&](const float4 *kk) -> float {
    float2 d = make_float2(0.0f, 0.0f);
#pragma unroll
    for (int i = 0; i < DH / 4; ++i) {
      d = fma2(make_float2(q[4 * i], q[4 * i + 1]), make_float2(kk[i].x, kk[i].y), d);
      d = fma2(make_float2(q[4 * i + 2], q[4 * i + 3]), make_float2(kk[i].z, kk[i].w), d);
    }
    return __fadd_rn(d.x, d.y);
  };
  // pass 1: scores and their maximum
  float mx = -INFINITY;
  for (int jb = 0; jb < nmax; jb += 8) {
    const uint4 w = (jb < cnt) ? __ldg(lst + (jb >> 3)) : make_uint4(0u, 0u, 0u, 0u);
    float sg[8];
#pragma unroll
    for (int k0 = 0; k0 < 8; k0 += U) {
      float4 kk[U][DH / 4];
#pragma unroll
      for (int k = 0; k < U; ++k) {
        const KeyRow<CLUSTER> kp = keyptr(idx_at(w, k0 + k));
#pragma unroll
        for (int i = 0; i < DH / 4; ++i) kk[k][i] = kp[i];
      }
#pragma unroll
      for (int k = 0; k < U; ++k) {
        sg[k0 + k] = __fmul_rn(dotk(kk[k]), scale);
        if (jb + k0 + k < cnt) mx = fmaxf(mx, sg[k0 + k]);
      }
    }
    if (jb < kRowCache) tmem_st<8>(tcache + jb, sg);
  }
  tmem_wait_st();
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
  for (int jb = 0; jb < nmax; jb += 8) {
    const uint4 w = (jb < cnt) ? __ldg(lst + (jb >> 3)) : make_uint4(0u, 0u, 0u, 0u);
    float sg[8];
    const bool cached = jb < kRowCache;
    if (cached) {
      tmem_ld<8>(tcache + jb, sg);
      tmem_wait_ld();
    }
#pragma unroll
    for (int k0 = 0; k0 < 8; k0 += U) {
      float4 vv[U][DH / 4];
#pragma unroll
      for (int k = 0; k < U; ++k) {
        const KeyRow<CLUSTER> kp = keyptr(idx_at(w, k0 + k));
        if (!cached) {
          float4 kk[DH / 4];
#pragma unroll
          for (int i = 0; i < DH / 4; ++i) kk[i] = kp[i];
          sg[k0 + k] = __fmul_rn(dotk(kk), scale);
        }
#pragma unroll
        for (int i = 0; i < DH / 4; ++i) vv[k][i] = kp[DH / 4 + i];
      }
      float pr[U];
#pragma unroll
      for (int k = 0; k < U; ++k) pr[k] = exp2_series(__fsub_rn(sg[k0 + k], mx));
#pragma unroll
      for (int k = 0; k < U; ++k)
        if (jb + k0 + k < cnt) accumulate(pr[k], vv[k]);
    }
  }
  const float inv = __fdiv_rn(1.0f, lsum);
#pragma unroll
  for (int i = 0; i < DH; ++i) A[i] = active ? __fmul_rn(num[i], inv) : 0.0f;
}

// byte k of a 16-entry index block
__device__ __forceinline__ int byte_at(const uint4 &w, int k) {
  const uint32_t v = k < 8 ? (k < 4 ? w.x : w.y) : (k < 12 ? w.z : w.w);
  return static_cast<int>((v >> (8 * (k & 3))) & 0xFFu);
}
// a 16-entry index block of consecutive rows r0, r0 + 1, ..., r0 + 15 (rows < 240, no byte carry)
__device__ __forceinline__ bool contiguous(const uint4 &w) {
  const uint32_t pat = (w.x & 0xFFu) * 0x01010101u + 0x03020100u;
  return w.x == pat && w.y == pat + 0x04040404u && w.z == pat + 0x08080808u && w.w == pat + 0x0C0C0C0Cu;
}

// One HPSA head for a query group (task mode).  Every lane walks the group's union key list in
// ascending token order; the loads are warp-uniform (shared-memory broadcasts).  A lane only
// folds in the keys of its own set (membership bit), so for each query the max, the sum l and
// the weighted sum num see exactly its keys, in ascending order, as in the canonical definition.
// Keys go two at a time through f32x2 instructions: the two lanes of a pair are independent
// computations, and the folds into l and num stay sequential in key order.
template <int DH, uint32_t STRIDE>
__device__ __forceinline__ void hpsa_task(const float *q, const uint4 mask, int cnt, const uint4 *ul,
                                          const uint8_t *rows, uint32_t kslot, float scale, uint32_t tcache,
                                          float *A) {
  auto kptr = [&](int off) { return reinterpret_cast<const float4 *>(rows + off * STRIDE + kslot); };
  // q . k (canonical order: even-feature and odd-feature FMA chains, then their sum); the two
  // chains are the two lanes of paired FMAs over adjacent features
  auto dot = [&](const float4 *k) -> float {
    float2 d = make_float2(0.0f, 0.0f);
#pragma unroll
    for (int i = 0; i < DH / 4; ++i) {
      d = fma2(make_float2(q[4 * i], q[4 * i + 1]), make_float2(k[i].x, k[i].y), d);
      d = fma2(make_float2(q[4 * i + 2], q[4 * i + 3]), make_float2(k[i].z, k[i].w), d);
    }
    return __fadd_rn(d.x, d.y);
  };
  auto dot2 = [&](const float4 *ka, const float4 *kb) -> float2 { return make_float2(dot(ka), dot(kb)); };
  const float2 sc = make_float2(scale, scale);
  constexpr int U = (DH >= 16) ? 2 : 4;  // keys per step (registers: U x d_h fp32 of K or V)
  // membership bits of a 16-key block (jb is a multiple of 16)
  auto segment = [&](int jb) -> uint32_t {
    const uint32_t word = jb < 64 ? (jb < 32 ? mask.x : mask.y) : (jb < 96 ? mask.z : mask.w);
    return word >> (jb & 16);
  };
  // pass 1: maximum score over the lane's keys.  The scores sigma = fl(dot * scale) of the first
  // kTaskCache keys also go to this warp's TMEM columns, so that pass 2 reads them back
  // instead of reloading K and recomputing the dot products (same values, bit for bit).
  float mx = -INFINITY;
  for (int jb = 0; jb < cnt; jb += 16) {
    const uint4 w = ul[jb >> 4];
    const uint32_t seg = segment(jb);
    const int nk = min(16, cnt - jb);
    float sgs[16];
    // the 16 keys of a full segment; DENSE: every lane holds all of them (no membership tests);
    // CONTIG: the keys are 16 consecutive rows (addresses at fixed offsets from the first)
    const bool contig = nk == 16 && contiguous(w);
    auto full_segment = [&](auto dense_tag, auto contig_tag) {
      constexpr bool DENSE = decltype(dense_tag)::value, CONTIG = decltype(contig_tag)::value;
#pragma unroll
      for (int k0 = 0; k0 < 16; k0 += U) {
        float4 kk[U][DH / 4];
#pragma unroll
        for (int k = 0; k < U; ++k) {
          const float4 *kp = CONTIG ? kptr(static_cast<int>(w.x & 0xFFu) + k0 + k) : kptr(byte_at(w, k0 + k));
#pragma unroll
          for (int i = 0; i < DH / 4; ++i) kk[k][i] = kp[i];
        }
#pragma unroll
        for (int k = 0; k < U; k += 2) {
          const float2 sg = mul2(dot2(kk[k], kk[k + 1]), sc);
          sgs[k0 + k] = sg.x, sgs[k0 + k + 1] = sg.y;
          if (DENSE || ((seg >> (k0 + k)) & 1u)) mx = fmaxf(mx, sg.x);
          if (DENSE || ((seg >> (k0 + k + 1)) & 1u)) mx = fmaxf(mx, sg.y);
        }
      }
    };
    if (nk == 16) {
      const bool dense = __all_sync(0xffffffffu, (seg & 0xFFFFu) == 0xFFFFu);
      if (contig) {
        if (dense) full_segment(std::true_type{}, std::true_type{});
        else full_segment(std::false_type{}, std::true_type{});
      } else {
        if (dense) full_segment(std::true_type{}, std::false_type{});
        else full_segment(std::false_type{}, std::false_type{});
      }
    } else {
#pragma unroll
      for (int k = 0; k < 16; k += 2) {
        if (k < nk) {
          const int k1 = (k + 1 < nk) ? k + 1 : k;
          float4 ka[DH / 4], kb[DH / 4];
          const float4 *pa = kptr(byte_at(w, k)), *pb = kptr(byte_at(w, k1));
#pragma unroll
          for (int i = 0; i < DH / 4; ++i) ka[i] = pa[i], kb[i] = pb[i];
          const float2 sg = mul2(dot2(ka, kb), sc);
          sgs[k] = sg.x, sgs[k + 1] = sg.y;
          if (((seg >> k) & 1u)) mx = fmaxf(mx, sg.x);
          if (k1 != k && ((seg >> k1) & 1u)) mx = fmaxf(mx, sg.y);
        } else {
          sgs[k] = 0.0f, sgs[k + 1] = 0.0f;
        }
      }
    }
    if (jb < kTaskCache) tmem_st<16>(tcache + jb, sgs);
  }
  tmem_wait_st();
  // pass 2: p = 2^(sigma - m), l += p, num += p v, in key order
  float lsum = 0.0f;
  float num[DH];
#pragma unroll
  for (int i = 0; i < DH; ++i) num[i] = 0.0f;
  // sigma - m for a pair of dot products (scalar: a product followed by a subtraction)
  auto shifted = [&](float2 d) {
    return make_float2(__fsub_rn(__fmul_rn(d.x, scale), mx), __fsub_rn(__fmul_rn(d.y, scale), mx));
  };
  auto fold = [&](float pr, const float4 *vv) {
    lsum = __fadd_rn(lsum, pr);
    const float2 pp = make_float2(pr, pr);
#pragma unroll
    for (int i = 0; i < DH / 4; ++i) {
      const float2 lo = fma2(pp, make_float2(vv[i].x, vv[i].y), make_float2(num[4 * i], num[4 * i + 1]));
      const float2 hi = fma2(pp, make_float2(vv[i].z, vv[i].w), make_float2(num[4 * i + 2], num[4 * i + 3]));
      num[4 * i] = lo.x, num[4 * i + 1] = lo.y, num[4 * i + 2] = hi.x, num[4 * i + 3] = hi.y;
    }
  };
  for (int jb = 0; jb < cnt; jb += 16) {
    const uint4 w = ul[jb >> 4];
    const uint32_t seg = segment(jb);
    const int nk = min(16, cnt - jb);
    if (jb < kTaskCache) {
      float sgs[16];
      tmem_ld<16>(tcache + jb, sgs);
      tmem_wait_ld();
      // DENSE: a full segment held by every lane (no membership or range tests); CONTIG: a full
      // segment of 16 consecutive rows
      auto cached_segment = [&](auto dense_tag, auto contig_tag) {
        constexpr bool DENSE = decltype(dense_tag)::value, CONTIG = decltype(contig_tag)::value;
#pragma unroll
        for (int k0 = 0; k0 < 16; k0 += U) {
          if (DENSE || CONTIG || k0 < nk) {
            float4 vv[U][DH / 4];
#pragma unroll
            for (int k = 0; k < U; ++k) {
              const float4 *kp = CONTIG ? kptr(static_cast<int>(w.x & 0xFFu) + k0 + k)
                                        : kptr(byte_at(w, DENSE ? k0 + k : min(k0 + k, nk - 1)));
#pragma unroll
              for (int i = 0; i < DH / 4; ++i) vv[k][i] = kp[DH / 4 + i];
            }
            float2 pr[U / 2];
#pragma unroll
            for (int k = 0; k < U; k += 2)
              // sigma - m for two keys: one paired add of -m (the cached scores are not products)
              pr[k / 2] = exp2_series2(add2(make_float2(sgs[k0 + k], sgs[k0 + k + 1]), make_float2(-mx, -mx)));
#pragma unroll
            for (int k = 0; k < U; k += 2) {
              if (DENSE || ((CONTIG || k0 + k < nk) && ((seg >> (k0 + k)) & 1u))) fold(pr[k / 2].x, vv[k]);
              if (DENSE || ((CONTIG || k0 + k + 1 < nk) && ((seg >> (k0 + k + 1)) & 1u)))
                fold(pr[k / 2].y, vv[k + 1]);
            }
          }
        }
      };
      const bool dense = nk == 16 && __all_sync(0xffffffffu, (seg & 0xFFFFu) == 0xFFFFu);
      if (nk == 16 && contiguous(w)) {
        if (dense) cached_segment(std::true_type{}, std::true_type{});
        else cached_segment(std::false_type{}, std::true_type{});
      } else {
        if (dense) cached_segment(std::true_type{}, std::false_type{});
        else cached_segment(std::false_type{}, std::false_type{});
      }
    } else if (nk == 16) {
#pragma unroll
      for (int k0 = 0; k0 < 16; k0 += U) {
        float4 kk[U][DH / 4], vv[U][DH / 4];
#pragma unroll
        for (int k = 0; k < U; ++k) {
          const float4 *kp = kptr(byte_at(w, k0 + k));
#pragma unroll
          for (int i = 0; i < DH / 4; ++i) kk[k][i] = kp[i];
#pragma unroll
          for (int i = 0; i < DH / 4; ++i) vv[k][i] = kp[DH / 4 + i];
        }
        float2 pr[U / 2];
#pragma unroll
        for (int k = 0; k < U; k += 2) pr[k / 2] = exp2_series2(shifted(dot2(kk[k], kk[k + 1])));
#pragma unroll
        for (int k = 0; k < U; k += 2) {
          if (((seg >> (k0 + k)) & 1u)) fold(pr[k / 2].x, vv[k]);
          if (((seg >> (k0 + k + 1)) & 1u)) fold(pr[k / 2].y, vv[k + 1]);
        }
      }
    } else {
      for (int k = 0; k < nk; k += 2) {
        const int k1 = (k + 1 < nk) ? k + 1 : k;
        float4 ka[DH / 4], kb[DH / 4], va[DH / 4], vb[DH / 4];
        const float4 *pa = kptr(byte_at(w, k)), *pb = kptr(byte_at(w, k1));
#pragma unroll
        for (int i = 0; i < DH / 4; ++i) ka[i] = pa[i], kb[i] = pb[i], va[i] = pa[DH / 4 + i], vb[i] = pb[DH / 4 + i];
        const float2 pr = exp2_series2(shifted(dot2(ka, kb)));
        if (((seg >> k) & 1u)) fold(pr.x, va);
        if (k1 != k && ((seg >> k1) & 1u)) fold(pr.y, vb);
      }
    }
  }
  const float inv = __fdiv_rn(1.0f, lsum);
#pragma unroll
  for (int i = 0; i < DH; ++i) A[i] = __fmul_rn(num[i], inv);
}

// ------------------------------------------------------------------------------------------
// weight streaming and tensor-core issue (run by warp 0 of each CTA)
// ------------------------------------------------------------------------------------------
// Chunk p of a block lives in stage p % S and completes phase parity (p / S) & 1 of full[stage]
// (and, D = 128, of empty[stage]); the operand-ready and accumulator-ready barriers complete one
// phase per GEMM, four per block, so GEMM g always waits for parity g & 1.  Everything the issue
// path computes is therefore a compile-time constant or a warp-uniform base address, and the
// tcgen05 instructions take their operands straight from uniform registers.
// What the issuer needs to know about the block a GEMM belongs to (used by the d = 128 schedule).
struct BlockCtx {
  uint32_t lpar;    // parity of the block's index in this CTA's sequence of blocks
  uint32_t kvf;     // cluster barrier: every CTA of the cluster has finished reading this CTA's K/V
  uint32_t kvf_ph;  // its phase parity for this block
  bool u_own;       // region U is this CTA's alone once its own attention is done (one-CTA cluster,
                    // or staged attention, whose peers read the K/V scratch in global memory)
};

template <int D, int ATT>
struct Issuer {
  using L = SmemLayout<D, ATT == 1>;
  using W = WeightSchedule<D>;
  static constexpr int S = W::kStages;
  static constexpr int CPL = W::kCPL;
  // some GEMM has more chunks than stages (D = 128): every chunk then releases its stage through
  // empty[stage], so that chunk p always completes phase parity (p / S) & 1 there
  static constexpr bool kRefillInGemm =
      W::count(0) > S || W::count(1) > S || W::count(2) > S || W::count(3) > S;
  uint32_t sb, tmem;
  Ctl ctl;
  uint32_t *n_issued;  // copies started so far (read by the teardown drain)

  // false once a wait of this CTA gave up: from then on nothing more is issued, so that the
  // teardown drain knows every copy and MMA in flight (only this warp's lane 0 sets the flag, in
  // a wait followed by __syncwarp, so every lane reads the same value)
  __device__ __forceinline__ bool live() const { return *ctl.abort == 0; }
  __device__ __forceinline__ void commit(uint32_t bar) const {
    if (live()) mma_commit_warp(bar);
  }
  __device__ __forceinline__ uint32_t bar_full(int s) const { return sb + L::kOffBar + 8 * s; }
  __device__ __forceinline__ uint32_t bar_empty(int s) const { return sb + L::kOffBar + 8 * (S + s); }
  __device__ __forceinline__ uint32_t bar_op() const { return sb + L::kOffBar + 16 * S; }
  __device__ __forceinline__ uint32_t bar_acc() const { return sb + L::kOffBar + 16 * S + 8; }
  // the accumulators are complete: let the CTA's other warps (waiting in wait_acc) go
  __device__ __forceinline__ static void release_acc() { named_bar_arrive(5, kEpiThreads); }

  // whole warp: lane 0 polls (the slow path is bounded and raises the abort flag), then the
  // warp reconverges
  __device__ __forceinline__ void wait(uint32_t bar, uint32_t parity) const {
    if ((threadIdx.x & 31) == 0 && !mbar_try_wait(bar, parity)) wait_bar_slow(ctl, bar, parity, false);
    __syncwarp();
  }
  // start the copy of chunk P of the block whose weights start at `src` (P is a template
  // parameter so that the chunk's geometry is evaluated at compile time)
  template <int P>
  __device__ __forceinline__ void copy(const uint8_t *src) const {
    constexpr ChunkDesc c = W::chunk(P);
    if (!live()) return;
    bulk_g2s_expect_warp(sb + L::kOffW + (P % S) * W::kStageBytes, src + c.off, c.bytes, bar_full(P % S));
    if ((threadIdx.x & 31) == 0) ++*n_issued;
  }
  // chunks 0 .. S-1 of the first block
  template <int P = 0>
  __device__ __forceinline__ void prologue(const uint8_t *w0) const {
    if constexpr (P < S) {
      copy<P>(w0);
      prologue<P + 1>(w0);
    }
  }
  // chunk J of GEMM G: (reuse a stage if the GEMM has more chunks than stages,) wait for the
  // weights, issue the MMAs over the chunk's K range, release the stage
  template <int G, int J>
  __device__ __forceinline__ void chunk_mmas(const uint8_t *w_cur) const {
    if constexpr (J < W::count(G)) {
      constexpr int p = W::first(G) + J;
      constexpr ChunkDesc c = W::chunk(p);
      constexpr uint32_t a_tile = (G == 3) ? L::kOffU : L::kOffAop;
      constexpr uint32_t a_sbo = (G == 3) ? (4u * D / 8u) * 128u : (D / 8u) * 128u;
      constexpr uint32_t b_sbo = (c.kcols / 8u) * 128u;
      constexpr uint32_t idesc = make_idesc_bf16(128, c.nrows);
      if constexpr (J >= S) {
        // reuse the stage of chunk p - S (same GEMM) once its MMAs are done
        wait(bar_empty((p - S) % S), ((p - S) / S) & 1);
        copy<p>(w_cur);
      }
      wait(bar_full(p % S), (p / S) & 1);
      const uint32_t b_tile = sb + L::kOffW + (p % S) * W::kStageBytes;
      if (live()) {
#pragma unroll 1
        for (int ks = 0; ks < c.kcols / 16; ++ks) {
          const uint32_t kabs = c.k0 + 16u * ks;
          mma_bf16_warp(tmem + c.n0, make_sdesc(sb + a_tile + (kabs / 8u) * 128u, 128u, a_sbo),
                        make_sdesc(b_tile + ks * 256u, 128u, b_sbo), idesc, kabs > 0 ? 1u : 0u);
        }
      }
      if constexpr (kRefillInGemm) commit(bar_empty(p % S));
      chunk_mmas<G, J + 1>(w_cur);
    }
  }
  // copies of chunks Q .. QEND-1 (positions past the block continue in the next block)
  template <int Q, int QEND>
  __device__ __forceinline__ void refill(const uint8_t *w_cur, const uint8_t *w_next, bool has_next) const {
    if constexpr (Q < QEND) {
      if constexpr (Q < CPL) copy<Q>(w_cur);
      else if (has_next) copy<Q - CPL>(w_next);
      refill<Q + 1, QEND>(w_cur, w_next, has_next);
    }
  }
  // Wait until every warp has published the operand of GEMM G, issue its tcgen05.mma chain
  // (accumulators at TMEM column 0), wait for its completion, then start the copies of the
  // chunks that follow the freed stages: chunk p + S of this block, or chunk p + S - CPL of the
  // next block (`w_next`, when `has_next`).
  template <int G>
  __device__ __forceinline__ void gemm(const uint8_t *w_cur, const uint8_t *w_next, bool has_next,
                                       const BlockCtx &) const {
    constexpr int first = W::first(G), count = W::count(G);
    wait(bar_op(), G & 1);
    tc_fence_after();
    chunk_mmas<G, 0>(w_cur);
    commit(bar_acc());
    // warp 0 alone waits for the accumulators; the other warps of the CTA wait in a named
    // barrier (no spinning), which warp 0 arrives at after the wait, before its copies
    wait(bar_acc(), G & 1);
    release_acc();
    // every MMA so far is complete, so the stages they read are free
    refill<(count > S ? first + count : first + S), first + count + S>(w_cur, w_next, has_next);
  }
  // every copy started has landed (bounded waits that ignore the abort flag)
  __device__ __forceinline__ void drain() const {
    const uint32_t n = *n_issued;
#pragma unroll
    for (int s = 0; s < S; ++s) {
      const uint32_t cnt = (n + S - 1 - s) / S;  // copies that went to stage s
      if (cnt > 0) wait_bar_drain(ctl, bar_full(s), (cnt - 1u) & 1u);
    }
  }
};
// d = 128: the 24 chunks of a block (16 KB each: QKV 0-5, O 6-7, FFN1 8-15, FFN2 16-23) do not
// fit three 16 KB stages without refilling inside the FFN GEMMs, so the schedule also uses the
// regions that are idle at that point of the block:
//   QKV  -> region U (free between the previous FFN2 and this block's K/V), one barrier bar_U;
//   O    -> stages W0, W1;
//   FFN1 -> region U again (free once every CTA of the cluster has finished attention);
//   FFN2 -> region U a third time, all eight chunks, copied during FFN1's epilogue as soon as
//           FFN1's MMAs (their last readers) are complete: FFN2's operand (the codes of u) is in
//           TMEM, columns [0, 256), and its accumulators in [256, 384), so no in-GEMM refill.
// Stage W2 and the operand-tile halves A0, A1 hold no weights (W2 holds the Q/A slots of tasks
// off their quadrant).  A barrier armed u times per block (u odd for U, W0, W1) completes phase
// parity (lpar if u is odd) ^ (index of the use within the block), with lpar the block's parity.
template <int ATT>
struct Issuer<128, ATT> {
  static constexpr int D = 128;
  using L = SmemLayout<D, ATT == 1>;
  using W = WeightSchedule<D>;
  static constexpr uint32_t kChunk = W::kStageBytes;
  static_assert(W::kCPL == 24 && W::kStages == 3 && kChunk == 16384, "d = 128 schedule");
  static_assert(L::kRegionU >= 8 * kChunk && L::kAopBytes == 2 * kChunk, "d = 128 regions");
  static constexpr uint32_t kFfn2Acc = 256;  // TMEM columns of FFN2's accumulators (codes of u in [0, 256))
  uint32_t sb, tmem;
  Ctl ctl;
  uint32_t *n_armed;  // [6] phases armed per weight barrier (W0, W1, W2, U, A0, A1), for the drain

  // barrier ids: 0-2 stages W0-W2, 3 region U, 4-5 operand-tile halves A0, A1
  __device__ __forceinline__ uint32_t bar(int id) const {
    return sb + L::kOffBar + (id < 3 ? 8 * id : 16 * 3 + 7 * 8 + 8 * (id - 3));
  }
  __device__ __forceinline__ uint32_t bar_empty(int s) const { return sb + L::kOffBar + 8 * (3 + s); }
  // false once a wait of this CTA gave up: nothing more is armed, copied or issued (see the
  // generic issuer)
  __device__ __forceinline__ bool live() const { return *ctl.abort == 0; }
  __device__ __forceinline__ void commit(uint32_t b) const {
    if (live()) mma_commit_warp(b);
  }
  __device__ __forceinline__ uint32_t bar_op() const { return sb + L::kOffBar + 48; }
  __device__ __forceinline__ uint32_t bar_acc() const { return sb + L::kOffBar + 56; }
  // FFN1's N tiles 0 and 1 (hidden units [0, 256)) are complete: once per block
  __device__ __forceinline__ uint32_t bar_acc_lo() const { return sb + L::kOffBar + 160; }
  // the accumulators are complete: let the CTA's other warps (waiting in wait_acc) go
  __device__ __forceinline__ static void release_acc() { named_bar_arrive(5, kEpiThreads); }

  // slot of chunk P: shared-memory offset, barrier id, uses of that barrier per block, use index
  struct Slot {
    uint32_t off;
    int id, uses, idx;
  };
  __host__ __device__ static constexpr Slot slot(int p) {
    return p < 6    ? Slot{L::kOffU + kChunk * p, 3, 3, 0}
           : p < 8  ? Slot{L::kOffW + kChunk * (p - 6), p - 6, 1, 0}
           : p < 16 ? Slot{L::kOffU + kChunk * (p - 8), 3, 3, 1}
                    : Slot{L::kOffU + kChunk * (p - 16), 3, 3, 2};
  }
  template <int P>
  __device__ __forceinline__ static uint32_t parity(uint32_t lpar) {
    constexpr Slot s = slot(P);
    return ((s.uses & 1) ? lpar : 0u) ^ static_cast<uint32_t>(s.idx & 1);
  }

  __device__ __forceinline__ void wait(uint32_t b, uint32_t parity, bool cluster_scope = false) const {
    if ((threadIdx.x & 31) == 0 && !(cluster_scope ? mbar_try_wait_acq_cluster(b, parity) : mbar_try_wait(b, parity)))
      wait_bar_slow(ctl, b, parity, cluster_scope);
    __syncwarp();
  }
  // arm barrier `id` for `bytes` (one arrive), then the copies of chunks P0 .. P1-1 complete it
  __device__ __forceinline__ void arm(int id, uint32_t bytes) const {
    if (!live()) return;
    asm volatile(
        "{\n\t.reg .pred e;\n\t.reg .b32 r;\n\telect.sync r|e, 0xffffffff;\n\t"
        "@e mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;\n\t}" ::"r"(bar(id)),
        "r"(bytes)
        : "memory");
    if ((threadIdx.x & 31) == 0) ++n_armed[id];
  }
  template <int P0, int P1>
  __device__ __forceinline__ void copies(const uint8_t *src) const {
    if (live()) copies_live<P0, P1>(src);
  }
  template <int P0, int P1>
  __device__ __forceinline__ void copies_live(const uint8_t *src) const {
    if constexpr (P0 < P1) {
      constexpr ChunkDesc c = W::chunk(P0);
      constexpr Slot s = slot(P0);
      asm volatile(
          "{\n\t.reg .pred e;\n\t.reg .b32 r;\n\telect.sync r|e, 0xffffffff;\n\t"
          "@e cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];\n\t}" ::"r"(
              sb + s.off),
          "l"(src + c.off), "r"(c.bytes), "r"(bar(s.id))
          : "memory");
      copies_live<P0 + 1, P1>(src);
    }
  }
  template <int P>
  __device__ __forceinline__ void copy1(const uint8_t *src) const {
    arm(slot(P).id, W::chunk(P).bytes);
    copies<P, P + 1>(src);
  }
  // QKV (region U) and O (W0, W1) of a block
  __device__ __forceinline__ void stage_qkv_o(const uint8_t *src) const {
    arm(3, 6 * kChunk);
    copies<0, 6>(src);
    copy1<6>(src);
    copy1<7>(src);
  }
  __device__ __forceinline__ void prologue(const uint8_t *w0) const { stage_qkv_o(w0); }
  // FFN2's eight chunks into region U.  Called by warp 0 during FFN1's epilogue once it has seen
  // FFN1's MMAs, the region's last readers in this block, complete.
  __device__ __forceinline__ void stage_ffn2(const uint8_t *w_cur) const {
    arm(3, 8 * kChunk);
    copies<16, 24>(w_cur);
  }

  // the MMAs of chunk P (its weights have landed)
  template <int G, int P>
  __device__ __forceinline__ void mmas() const {
    constexpr ChunkDesc c = W::chunk(P);
    constexpr uint32_t a_tile = (G == 3) ? L::kOffU : L::kOffAop;
    constexpr uint32_t a_sbo = (G == 3) ? (4u * D / 8u) * 128u : (D / 8u) * 128u;
    constexpr uint32_t b_sbo = (c.kcols / 8u) * 128u;
    constexpr uint32_t idesc = make_idesc_bf16(128, c.nrows);
    const uint32_t b_tile = sb + slot(P).off;
    if (!live()) return;
#pragma unroll 1
    for (int ks = 0; ks < c.kcols / 16; ++ks) {
      const uint32_t kabs = c.k0 + 16u * ks;
      mma_bf16_warp(tmem + c.n0, make_sdesc(sb + a_tile + (kabs / 8u) * 128u, 128u, a_sbo),
                    make_sdesc(b_tile + ks * 256u, 128u, b_sbo), idesc, kabs > 0 ? 1u : 0u);
    }
  }
  // the MMAs of chunks P and P + 1, two 128-row N tiles of one K range that sit next to each other
  // in shared memory, as N = 256 MMAs (the tensor pipe runs an N = 256 MMA at close to its peak,
  // two N = 128 ones at about 60% of it)
  template <int G, int P>
  __device__ __forceinline__ void mmas_pair() const {
    constexpr ChunkDesc c = W::chunk(P), c2 = W::chunk(P + 1);
    static_assert(c.nrows == 128 && c2.nrows == 128 && c2.n0 == c.n0 + 128 && c2.k0 == c.k0 &&
                      c2.kcols == c.kcols && slot(P + 1).off == slot(P).off + kChunk,
                  "an N-tile pair: adjacent tiles of one K range");
    constexpr uint32_t a_tile = (G == 3) ? L::kOffU : L::kOffAop;
    constexpr uint32_t a_sbo = (G == 3) ? (4u * D / 8u) * 128u : (D / 8u) * 128u;
    constexpr uint32_t b_sbo = (c.kcols / 8u) * 128u;  // row groups 16..31 continue in chunk P + 1
    constexpr uint32_t idesc = make_idesc_bf16(128, 256);
    const uint32_t b_tile = sb + slot(P).off;
    if (!live()) return;
#pragma unroll 1
    for (int ks = 0; ks < c.kcols / 16; ++ks) {
      const uint32_t kabs = c.k0 + 16u * ks;
      mma_bf16_warp(tmem + c.n0, make_sdesc(sb + a_tile + (kabs / 8u) * 128u, 128u, a_sbo),
                    make_sdesc(b_tile + ks * 256u, 128u, b_sbo), idesc, kabs > 0 ? 1u : 0u);
    }
  }

  // FFN2 chunk P: A (the codes of u) from TMEM, K element k of a row in column k / 2; the
  // accumulators in columns [kFfn2Acc, kFfn2Acc + 128)
  template <int P>
  __device__ __forceinline__ void mmas_tmem_a() const {
    constexpr ChunkDesc c = W::chunk(P);
    static_assert(c.gemm == 3 && c.n0 == 0 && c.nrows == 128, "an FFN2 chunk");
    constexpr uint32_t b_sbo = (c.kcols / 8u) * 128u;
    constexpr uint32_t idesc = make_idesc_bf16(128, c.nrows);
    const uint32_t b_tile = sb + slot(P).off;
    if (!live()) return;
#pragma unroll 1
    for (int ks = 0; ks < c.kcols / 16; ++ks) {
      const uint32_t kabs = c.k0 + 16u * ks;
      mma_bf16_tmem_a_warp(tmem + kFfn2Acc, tmem + kabs / 2u, make_sdesc(b_tile + ks * 256u, 128u, b_sbo), idesc,
                           kabs > 0 ? 1u : 0u);
    }
  }

  template <int G>
  __device__ __forceinline__ void gemm(const uint8_t *w_cur, const uint8_t *w_next, bool has_next,
                                       const BlockCtx &bc) const {
    const uint32_t lp = bc.lpar;
    wait(bar_op(), G & 1);
    tc_fence_after();
    if constexpr (G == 0) {
      wait(bar(3), parity<0>(lp));  // QKV weights in region U
      mmas_pair<0, 0>();  // N tiles 0 and 1, K 0..63
      mmas_pair<0, 2>();  // N tiles 0 and 1, K 64..127
      mmas<0, 4>();       // N tile 2
      mmas<0, 5>();
      commit(bar_acc());
      wait(bar_acc(), 0);
      release_acc();
    } else if constexpr (G == 1) {
      wait(bar(0), parity<6>(lp));
      mmas<1, 6>();
      wait(bar(1), parity<7>(lp));
      mmas<1, 7>();
      commit(bar_acc());
      // FFN1 weights into region U: this CTA has finished reading it (every warp published the O
      // operand) and no peer reads it (one-CTA cluster, staged attention); a cluster whose peers
      // read this CTA's K/V stages them at FFN1 instead, so that the O epilogue overlaps the
      // peers' attention.
      if (bc.u_own) {
        arm(3, 8 * kChunk);
        copies<8, 16>(w_cur);
      }
      wait(bar_acc(), 1);
      release_acc();
    } else if constexpr (G == 2) {
      if (!bc.u_own) {  // every CTA of the cluster is done with this CTA's K/V
        wait(bc.kvf, bc.kvf_ph, true);
        arm(3, 8 * kChunk);
        copies<8, 16>(w_cur);
      }
      wait(bar(3), parity<8>(lp));  // FFN1 weights in region U
      mmas_pair<2, 8>();
      mmas_pair<2, 10>();
      // the epilogue of accumulator columns [0, 256), the first half of every column slice's hidden
      // units, starts while the MMAs of [256, 512) run (every warp waits on both barriers itself;
      // no release by this warp)
      commit(bar_acc_lo());
      mmas_pair<2, 12>();
      mmas_pair<2, 14>();
      commit(bar_acc());
    } else {
      // all eight chunks in region U (copied during FFN1's epilogue); A from TMEM
      wait(bar(3), parity<16>(lp));
      mmas_tmem_a<16>();
      mmas_tmem_a<17>();
      mmas_tmem_a<18>();
      mmas_tmem_a<19>();
      mmas_tmem_a<20>();
      mmas_tmem_a<21>();
      mmas_tmem_a<22>();
      mmas_tmem_a<23>();
      commit(bar_acc());
      wait(bar_acc(), 1);
      release_acc();
      if (has_next) stage_qkv_o(w_next);  // region U and W0, W1 are free again
    }
  }
  // every copy started has landed (bounded waits that ignore the abort flag)
  __device__ __forceinline__ void drain() const {
#pragma unroll
    for (int id = 0; id < 6; ++id) {
      const uint32_t cnt = n_armed[id];
      if (cnt > 0) wait_bar_drain(ctl, bar(id), (cnt - 1u) & 1u);
    }
  }
};

// ------------------------------------------------------------------------------------------
// the kernel
// ------------------------------------------------------------------------------------------
template <int D, int ATT, int ACT, int LIN>
__global__ void __launch_bounds__(kThreads, 1) aecct_decoder_kernel(const __grid_constant__ DecodeParams p) {
  // ATT: 0 = per-row neighbour lists, 1 = warp tasks, 2 = per-row lists over per-head staged rows
  constexpr bool TASKS = ATT == 1, STAGED = ATT == 2;
  static_assert(!STAGED || D == 128, "staged attention is built for d = 128");
  using L = SmemLayout<D, TASKS>;
  using LP = LayerParamLayout;
  constexpr int DH = D / kHeads;  // head width
  constexpr int XS = D / 4;       // x columns per thread
  // the O and FFN2 biases are loaded before the accumulator waits where the registers allow it
  // (d <= 64; at d = 128 the 32 extra live registers spill)
  constexpr bool kEarlyBias = D <= 64;
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
  uint32_t *s_kvcl = reinterpret_cast<uint32_t *>(smem + L::kOffMisc + 8);   // [8] shared::cluster K/V bases per CTA
  uint64_t *s_zgen = reinterpret_cast<uint64_t *>(smem + L::kOffMisc + 72);   // [8] generic z bases per CTA
  uint32_t *s_issued = reinterpret_cast<uint32_t *>(smem + L::kOffMisc + 136);  // [10] weight copies / phases armed
  // staged attention: warps past their reads of a buffer set in the current head round ([2] sets)
  uint32_t *s_headdone = reinterpret_cast<uint32_t *>(smem + L::kOffMisc + 176);
  // staged attention: the barriers of the K and V buffers (buffer set 0; set 1 when two heads fit)
  const uint32_t bar_sk = bar_fin + 32, bar_sv = bar_fin + 40;  // + 16: set 1

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
    if constexpr (D == 128)  // region U, the two operand-tile halves (d = 128 weight schedule), the
                             // staged K/V buffers, FFN1's first half
      for (int i = 0; i < 8; ++i) mbar_init(bar_fin + 8 + 8 * i, 1);
    *s_abort = 0;
    for (int i = 0; i < 10; ++i) s_issued[i] = 0;
    s_headdone[0] = s_headdone[1] = 0;
    // base of the K/V area of every CTA of the cluster as a shared::cluster address, and generic
    // base of its z area: this CTA's own through its plain shared-memory window, the others
    // through the distributed shared window
    for (int c = 0; c < p.C; ++c) {
      const bool own = c == static_cast<int>(crank);
      s_kvcl[c] = mapa_cluster(smem_u32(smem + L::kOffU), c);
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
  // the attention plan, into shared memory (read by every task of every block); the first CTA-wide
  // barrier of the group loop orders it before its readers
  uint8_t *const splan = smem + L::kTotal;
  for (uint32_t i = threadIdx.x; i < p.plan_bytes / 16u; i += kThreads)
    reinterpret_cast<uint4 *>(splan)[i] = __ldg(p.plan_blob + i);

  const Issuer<D, ATT> issuer{sb, tmem, ctl, s_issued};
  if (warp == 0 && cluster_id < p.n_groups) issuer.prologue(p.wstream);
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
    uint32_t *bitw = reinterpret_cast<uint32_t *>(smem + L::kOffBitWords);  // [G][hwords] bitmasks
    const int W = p.hwords;
    const uint32_t qbar = 1 + qd;  // named barrier of the 4 warps sharing a lane quadrant
    // d = 128 warp tasks run off their rows' quadrant: the Q/A slots (2 KB: 32 rows of 16 floats,
    // 16-byte piece f of row i at f ^ ((i >> 1) & 3)) in weight stage W2, idle from the previous
    // block's FFN2 to this block's O GEMM; the plan's table gives each quadrant's group and each
    // (group, head)'s slot (0xFF: none)
    const uint8_t *qtab = splan + p.off_qslot;
    const uint32_t qslot_base = sb + L::kOffW + 2u * WeightSchedule<D>::kStageBytes;
    static_assert(D != 128 || kQSlots * 2048u <= WeightSchedule<D>::kStageBytes, "the Q/A slots fit W2");
    auto qslot_piece = [&](uint32_t slot, int i, int f) -> uint32_t {
      return qslot_base + slot * 2048u + static_cast<uint32_t>(i) * 64u + static_cast<uint32_t>((f ^ ((i >> 1) & 3)) << 4);
    };
    const int T = p.T, Tp = p.Tp, n = p.n, m = p.m, de = D - p.d_spe;
    const int W4 = 4 * D;
    const float inv_d = 1.0f / static_cast<float>(D);
    uint32_t kvr_ph = 0, kvf_ph = 0, zr_ph = 0, zf_ph = 0;
    int64_t z_uses = 0;

    // reduce one value per row over the 4 slices: max or pairwise sum ((s0+s1)+(s2+s3))
    auto row_max = [&](float v) -> float {
      *red.slot(sl, r) = v;
      named_bar_sync(qbar, 128);
      const float a = fmaxf(fmaxf(*red.slot(0, r), *red.slot(1, r)), fmaxf(*red.slot(2, r), *red.slot(3, r)));
      red.sel ^= 1;
      return a;
    };
    // Per-word alpha (alpha_mode 1, one CTA per word): the max of the row absmaxes over the rows
    // of this row's codeword, through the z area (free until S9) and the bitmask area (free
    // between the group start and S10).  Word g's rows are [g T, g T + T).
    float *rowmax_s = reinterpret_cast<float *>(smem + L::kOffZ);
    float *wordmax_s = reinterpret_cast<float *>(smem + L::kOffBitWords);
    auto word_alpha = [&](float a_row) -> float {
      if (p.alpha_mode == 0) return a_row;
      if (sl == 0) rowmax_s[r] = a_row;
      named_bar_sync(5, kEpiThreads);
      if (warp < p.G) {
        float a = 0.0f;
        for (int i = lane; i < p.Tp; i += 32) a = fmaxf(a, rowmax_s[warp * p.Tp + i]);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) a = fmaxf(a, __shfl_xor_sync(0xffffffffu, a, o));
        if (lane == 0) wordmax_s[warp] = a;
      }
      named_bar_sync(5, kEpiThreads);
      const int gw = (static_cast<int>(crank) * kRows + r) / p.Tp;
      return gw < p.G ? wordmax_s[gw] : a_row;
    };
    auto row_sum = [&](float v) -> float {
      *red.slot(sl, r) = v;
      named_bar_sync(qbar, 128);
      const float a = __fadd_rn(__fadd_rn(*red.slot(0, r), *red.slot(1, r)), __fadd_rn(*red.slot(2, r), *red.slot(3, r)));
      red.sel ^= 1;
      return a;
    };
    // publish this warp's part of the operand of GEMM `gemm` of block `blk` of group `gi`;
    // warp 0 then issues the GEMM and prefetches the weights that follow it
    uint32_t blk_base = 0;  // blocks this CTA ran in earlier groups (the block parity of the d = 128 schedule)
    auto signal_op = [&](int gemm, int blk, int64_t gi) {
      tc_fence_before();  // this thread's TMEM reads are ordered before the MMA the arrive releases
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(bar_op);
      __syncwarp();
      if (warp == 0) {
        const bool last_blk = blk + 1 == p.n_layers;
        const uint8_t *w_cur = p.wstream + static_cast<size_t>(blk) * p.layer_bytes;
        const uint8_t *w_next = last_blk ? p.wstream : w_cur + p.layer_bytes;
        const bool has_next = !last_blk || gi + p.n_clusters < p.n_groups;
        const BlockCtx bc{(blk_base + static_cast<uint32_t>(blk)) & 1u, bar_kvf, kvf_ph, p.C == 1 || STAGED};
        if (gemm == 0) issuer.template gemm<0>(w_cur, w_next, has_next, bc);
        if (gemm == 1) issuer.template gemm<1>(w_cur, w_next, has_next, bc);
        if (gemm == 2) issuer.template gemm<2>(w_cur, w_next, has_next, bc);
        if (gemm == 3) issuer.template gemm<3>(w_cur, w_next, has_next, bc);
      }
    };
    // A cluster of one CTA needs no cluster-scope signal: the named barrier in cluster_arrive
    // already orders every access of the CTA, so cluster_wait has nothing left to wait for.
    auto cluster_arrive = [&](uint32_t bar) {
      // all 512 CUDA-core threads of this CTA are past their accesses: tell every CTA
      named_bar_sync(5, kEpiThreads);
      if (p.C == 1) return;
      if (tid == 0) {
        fence_acq_rel_cluster();
        for (int c = 0; c < p.C; ++c) mbar_arrive_cluster(mapa_cluster(bar, c));
      }
      __syncwarp();
    };
    // after a CTA-wide barrier: this CTA no longer reads any CTA's K/V of this block (signalled by
    // thread `who`)
    auto kvf_signal = [&](int who) {
      if (p.C == 1) return;
      if (tid == who) {
        fence_acq_rel_cluster();
        for (int c = 0; c < p.C; ++c) mbar_arrive_cluster(mapa_cluster(bar_kvf, c));
      }
      __syncwarp();
    };
    // accumulators of the last GEMM are complete once warp 0, which waited for them in its
    // gemm<G> call and then arrived at this barrier, releases it
    auto wait_acc = [&]() {
      if (warp != 0) named_bar_sync(5, kEpiThreads);
      tc_fence_after();
    };
    // wait for a cluster-wide phase: thread 0 waits on the mbarrier, the others in a named barrier
    auto cluster_wait = [&](uint32_t bar, uint32_t &ph) {
      if (p.C == 1) return;
      if (tid == 0) wait_bar(ctl, bar, ph, true);
      ph ^= 1u;
      __syncwarp();
      named_bar_sync(5, kEpiThreads);
    };

    for (int64_t gi = cluster_id; gi < p.n_groups; gi += p.n_clusters) {
      // the group's channel outputs, in one coalesced pass, into the decoded-bits area (free
      // until S10; G n < C x 128 floats fit); the next group's are prefetched into L2
      float *ybuf = reinterpret_cast<float *>(obits);
      {
        const int64_t y0 = gi * p.G * n;
        const int64_t ny = min(static_cast<int64_t>(p.G) * n, p.B * n - y0);
        for (int i = tid; i < ny; i += kEpiThreads) ybuf[i] = __ldg(p.y + y0 + i);
        const int64_t y1 = y0 + static_cast<int64_t>(p.n_clusters) * p.G * n;
        const int64_t ny1 = min(static_cast<int64_t>(p.G) * n, p.B * n - y1);
        for (int64_t i = static_cast<int64_t>(tid) * 32; i < ny1; i += kEpiThreads * 32)
          asm volatile("prefetch.global.L2 [%0];" ::"l"(p.y + y1 + i));
      }
      if (named_bar_or(5, kEpiThreads, *s_abort != 0)) break;
      // hard decisions of the group's words as bitmasks (one warp ballot per 32 variables)
      for (int wi = warp; wi < p.G * W; wi += kEpiWarps) {
        const int gw = wi / W, j = 32 * (wi - gw * W) + lane;
        const bool neg = j < n && gi * p.G + gw < p.B && ybuf[gw * n + j] < 0.0f;
        const uint32_t word = __ballot_sync(0xffffffffu, neg);
        if (lane == 0) bitw[wi] = word;
      }
      named_bar_sync(5, kEpiThreads);
      const int rho = static_cast<int>(crank) * kRows + r;
      const int g = rho / Tp;
      const int t = __ldg(p.perm + (rho - g * Tp));  // token held by this row (0xFFFF: a padding row)
      const int64_t b = gi * p.G + g;
      const bool row_cw = g < p.G && t != 0xFFFF;
      const bool valid = row_cw && b < p.B;
      const bool cap = valid && b < p.cap_B;
      const float *yrow = ybuf + (valid ? g : 0) * n;

      float x[XS];
      float alpha_in;
      // ---------------- S1/S2: tokens, embedding, SPE (Sec. 3, Sec. 4.3)
      {
        float h = 0.0f;
        if (valid) {
          if (t < n) {
            h = fabsf(yrow[t]);
          } else {
            const int i = t - n;
            // s_i = parity of H_i AND b(y) (Sec. 3), over the bitmask words
            uint32_t par = 0;
            for (int w = 0; w < W; ++w) par += __popc(__ldg(p.hbits + i * W + w) & bitw[g * W + w]);
            par &= 1u;
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
      // Quant(x) -> QKV operand (Sec. 4.1 eq. Quant); full-precision linears: x rounded to bf16
      auto quant_x_to_aop = [&]() -> float {
        if constexpr (LIN == 1) {
          store_bf16<XS>(aop, r, sl * XS, D, x);
          return 0.0f;
        }
        float a = 0.0f;
#pragma unroll
        for (int j = 0; j < XS; ++j) a = fmaxf(a, fabsf(x[j]));
        a = word_alpha(row_max(a));
        a = (a > p.alpha_floor) ? a : p.alpha_floor;
        alpha_in = a;
        const float rr = __fdiv_rn(127.0f, a);
        float qv[XS];
        codes<XS>(x, rr, qv);
        store_codes<XS>(aop, r, sl * XS, D, qv);
        return rr;
      };
      // dequantisation factor gamma*delta * alpha / Q_b of eq. AAPLinear for the scale at swp;
      // 1 for full-precision linears (out = acc + b)
      auto dq_factor = [&](const float *swp) -> float {
        if constexpr (LIN == 1) return 1.0f;
        return __fdiv_rn(__fmul_rn(__ldg(swp), alpha_in), 127.0f);
      };
      // x <- LayerNorm(x + (acc * f + bias)) with gamma g and beta be (Post-LN, Sec. 5)
      auto residual_ln = [&](const float *ac, float f, const float *bb, const float *g, const float *be) {
        float v[XS];
        dequant<XS>(ac, f, bb, v);
#pragma unroll
        for (int j = 0; j < XS; ++j) v[j] = __fadd_rn(x[j], v[j]);
        const float mu = __fmul_rn(row_sum(psum<XS>(v)), inv_d);
        float sq[XS];
#pragma unroll
        for (int j = 0; j < XS; ++j) {
          v[j] = __fsub_rn(v[j], mu);
          sq[j] = __fmul_rn(v[j], v[j]);
        }
        const float var = __fmul_rn(row_sum(psum<XS>(sq)), inv_d);
        const float rstd = __fdiv_rn(1.0f, __fsqrt_rn(__fadd_rn(var, p.ln_eps)));
        float gg[XS], bt[XS];
        ldg_vec<XS>(g, gg);
        ldg_vec<XS>(be, bt);
#pragma unroll
        for (int j = 0; j < XS; ++j) x[j] = __fadd_rn(__fmul_rn(__fmul_rn(v[j], rstd), gg[j]), bt[j]);
      };
      auto capture_q = [&](int layer, int gemm, const float *qv, int c0, int len, float alpha) {
        if constexpr (LIN == 1) return;  // no codes or alpha with full-precision linears
        const int64_t row = ((b * p.n_layers + layer) * 4 + gemm) * T + t;
        if (p.cap_q)
          for (int j = 0; j < len; ++j) p.cap_q[row * W4 + c0 + j] = static_cast<int8_t>(qv[j]);
        if (p.cap_alpha && sl == 0) p.cap_alpha[row] = alpha;
      };
      auto capture_acc = [&](int layer, int gemm, const float *av, int c0, int len) {
        const int64_t row = ((b * p.n_layers + layer) * 4 + gemm) * T + t;
        if (p.cap_acc)
          for (int j = 0; j < len; ++j)
            p.cap_acc[row * W4 + c0 + j] = LIN == 1 ? __float_as_int(av[j]) : static_cast<int32_t>(av[j]);
      };

      {
        const float rr = quant_x_to_aop();
        if (cap) {
          float qv[XS];
          codes<XS>(x, rr, qv);
          capture_q(0, 0, qv, sl * XS, XS, alpha_in);
        }
      }
      signal_op(0, 0, gi);

      for (int l = 0; l < p.n_layers; ++l) {
        const float *lp = p.lparams + (size_t)l * LP::stride(D);
        const float *sw = lp + LP::sw(D);
        // ---------------- S4 epilogue: K, V to shared memory
        const float fq = dq_factor(sw + 0);
        const float fk = dq_factor(sw + 1);
        const float fv = dq_factor(sw + 2);
        wait_acc();
        // park the residual row in TMEM columns [3D, 4D) (unused by the QKV and O accumulators)
        // so that attention runs with the registers it needs
        tmem_st<XS>(tl + 3 * D + sl * XS, x);
        tmem_wait_st();
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
          const int e = sl + 4 * hh;
          float ka[DH], va[DH], bk[DH], bv[DH];
          ldg_vec<DH>(lp + LP::bqkv(D) + D + e * DH, bk);
          ldg_vec<DH>(lp + LP::bqkv(D) + 2 * D + e * DH, bv);
          tmem_ld<DH>(tl + D + e * DH, ka);
          tmem_ld<DH>(tl + 2 * D + e * DH, va);
          tmem_wait_ld();
          if (cap) {
            capture_acc(l, 0, ka, D + e * DH, DH);
            capture_acc(l, 0, va, 2 * D + e * DH, DH);
          }
          dequant<DH>(ka, fk, bk, ka);
          dequant<DH>(va, fv, bv, va);
          if constexpr (STAGED) {
            // K and V of this row and head, head-major in region U ([head][K, V][128 rows][64 B],
            // 16-byte piece f of row r at f ^ ((r >> 1) & 3)): the layout of the cluster's scratch
            // in global memory, where bulk copies take them next
            const uint32_t kd = kvl + ((static_cast<uint32_t>(e) * 2u) * kRows + r) * 64u;
            const uint32_t vd = kd + kRows * 64u;
#pragma unroll
            for (int f = 0; f < DH / 4; ++f) {
              const uint32_t g = static_cast<uint32_t>((f ^ ((r >> 1) & 3)) << 4);
              st_shared_f4(kd + g, ka[4 * f], ka[4 * f + 1], ka[4 * f + 2], ka[4 * f + 3]);
              st_shared_f4(vd + g, va[4 * f], va[4 * f + 1], va[4 * f + 2], va[4 * f + 3]);
            }
          } else {
            // head slot of this row: (K | V), or (Q | K | V) in task mode at d <= 64
            const uint32_t dst = kvl + r * L::kKvStride + e * L::kSlot + (L::kQInSmem ? 4 * DH : 0);
#pragma unroll
            for (int i = 0; i < DH; i += 4) {
              st_shared_f4(dst + 4 * i, ka[i], ka[i + 1], ka[i + 2], ka[i + 3]);
              st_shared_f4(dst + 4 * (DH + i), va[i], va[i + 1], va[i + 2], va[i + 3]);
            }
          }
          if constexpr (L::kQInSmem) {
            float qa[DH], bq[DH];
            ldg_vec<DH>(lp + LP::bqkv(D) + e * DH, bq);
            tmem_ld<DH>(tl + e * DH, qa);
            tmem_wait_ld();
            if (cap) capture_acc(l, 0, qa, e * DH, DH);
            const uint32_t qdst = kvl + r * L::kKvStride + e * L::kSlot;
            dequant<DH>(qa, fq, bq, qa);
#pragma unroll
            for (int i = 0; i < DH; i += 4) st_shared_f4(qdst + 4 * i, qa[i], qa[i + 1], qa[i + 2], qa[i + 3]);
          } else if constexpr (TASKS) {
            // this row's Q of head e into the slot of a task (group, e) that runs off this quadrant
            const uint32_t qg = qtab[qd];
            const uint32_t qs = qg != 0xFFu ? qtab[4 + qg * 8 + e] : 0xFFu;
            if (qs != 0xFFu) {
              float qa[DH], bq[DH];
              ldg_vec<DH>(lp + LP::bqkv(D) + e * DH, bq);
              tmem_ld<DH>(tl + e * DH, qa);
              tmem_wait_ld();
              if (cap) capture_acc(l, 0, qa, e * DH, DH);
              dequant<DH>(qa, fq, bq, qa);
#pragma unroll
              for (int f = 0; f < DH / 4; ++f)
                st_shared_f4(qslot_piece(qs, lane, f), qa[4 * f], qa[4 * f + 1], qa[4 * f + 2], qa[4 * f + 3]);
            }
          }
        }
        if constexpr (TASKS) {
          // ---------------- S5: HPSA (Sec. 4.2), task mode: warp tasks over query groups
          named_bar_sync(5, kEpiThreads);  // every Q, K, V row of this CTA is in shared memory
          // this warp's score cache: its lane quadrant, kTaskCache columns from kTaskCacheCol
          static_assert(L::kQInSmem ? (L::kTaskCacheCol >= 4u * D && L::kTaskCacheCol + 4u * kTaskCache <= L::kTmemCols)
                                    : (L::kTaskCacheCol >= 1u * D && L::kTaskCacheCol + 4u * kTaskCache <= 3u * D),
                        "TMEM: the cache clears Q/A, the live accumulators and the parked residual");
          // d = 128: a task's 32 rows are this warp's TMEM lane quadrant (the plan keeps every task on
          // a warp of its group's quadrant); Q comes from the QKV accumulators of this thread's row
          // and the output goes back over them
          const uint32_t tcache = tmem + (static_cast<uint32_t>(32 * (warp & 3)) << 16) + L::kTaskCacheCol +
                                  static_cast<uint32_t>(warp >> 2) * kTaskCache;
          for (int k = 0; k < kMaxTasks; ++k) {
            const uint32_t task = reinterpret_cast<const uint16_t *>(splan + p.off_task)[warp * kMaxTasks + k];
            if (task == 0xFFFFu) break;
            const int grp = static_cast<int>(task >> 3), e = static_cast<int>(task & 7u);
            const int ring = e < p.h_first ? 0 : 1;
            const uint4 gi = reinterpret_cast<const uint4 *>(splan + p.off_grp)[grp];
            const bool act = lane < static_cast<int>(gi.y);
            const int row = static_cast<int>(gi.x) + (act ? lane : 0);
            // a lane past the group's rows computes on row 0 and its result is dropped; an all-ones
            // mask keeps it from breaking the dense fast path
            const uint4 mk = act ? reinterpret_cast<const uint4 *>(splan + p.off_mask)[(grp * 2 + ring) * 32 + lane]
                                 : make_uint4(~0u, ~0u, ~0u, ~0u);
            const uint32_t ui = reinterpret_cast<const uint32_t *>(splan + p.off_uinfo)[grp * 2 + ring];
            float q[DH], a[DH];
            // d = 128: a task off its rows' quadrant has Q and A in a W2 slot (row = lane)
            const uint32_t qs = L::kQInSmem ? 0xFFu : qtab[4 + grp * 8 + e];
            if constexpr (L::kQInSmem) {
              const float4 *qp = reinterpret_cast<const float4 *>(smem + L::kOffU + row * L::kKvStride + e * L::kSlot);
#pragma unroll
              for (int i = 0; i < DH / 4; ++i) {
                const float4 v = qp[i];
                q[4 * i] = v.x, q[4 * i + 1] = v.y, q[4 * i + 2] = v.z, q[4 * i + 3] = v.w;
              }
            } else if (qs != 0xFFu) {
#pragma unroll
              for (int f = 0; f < DH / 4; ++f) {
                const float4 v = ld_shared_f4(qslot_piece(qs, lane, f));
                q[4 * f] = v.x, q[4 * f + 1] = v.y, q[4 * f + 2] = v.z, q[4 * f + 3] = v.w;
              }
            } else {
              float qa[DH], bq[DH];
              ldg_vec<DH>(lp + LP::bqkv(D) + e * DH, bq);
              tmem_ld<DH>(tl + e * DH, qa);
              tmem_wait_ld();
              if (cap) capture_acc(l, 0, qa, e * DH, DH);
              dequant<DH>(qa, fq, bq, q);
            }
            hpsa_task<DH, L::kKvStride>(q, mk, static_cast<int>(ui & 255u),
                                        reinterpret_cast<const uint4 *>(splan + p.off_ulist) + (ui >> 8),
                                        smem + L::kOffU + gi.z * L::kKvStride,
                                        e * L::kSlot + (L::kQInSmem ? 4 * DH : 0), p.att_scale, tcache, a);
            if constexpr (L::kQInSmem) {
              if (act) {
                // A of (row, head e) replaces Q of (row, head e): this task was its only reader
                float4 *ap = reinterpret_cast<float4 *>(smem + L::kOffU + row * L::kKvStride + e * L::kSlot);
#pragma unroll
                for (int i = 0; i < DH / 4; ++i) ap[i] = make_float4(a[4 * i], a[4 * i + 1], a[4 * i + 2], a[4 * i + 3]);
              }
            } else if (qs != 0xFFu) {
              // A of (row, head e) over its Q in the slot (this task was its only reader)
#pragma unroll
              for (int f = 0; f < DH / 4; ++f) st_shared_f4(qslot_piece(qs, lane, f), a[4 * f], a[4 * f + 1], a[4 * f + 2], a[4 * f + 3]);
            } else {
              // every lane's own row: A of (row, head e) over the head's Q accumulators (a lane past
              // the group's rows writes a padding or empty row, which nothing reads)
              tmem_st<DH>(tl + e * DH, a);
            }
            __syncwarp();
          }
          if constexpr (!L::kQInSmem) {
            tmem_wait_st();
            tc_fence_before();  // the TMEM stores are ordered before the barrier for the row owners
          }
          named_bar_sync(5, kEpiThreads);  // A complete; Q, K, V no longer read
          // Quant(A) -> O operand, by row slices
          // columns [sl XS, sl XS + XS) are heads 2 sl and 2 sl + 1, in their Q slots (shared memory)
          // or over their Q accumulators (TMEM, d = 128)
          float av[XS];
          if constexpr (L::kQInSmem) {
#pragma unroll
            for (int hh = 0; hh < 2; ++hh) {
              const float4 *ap =
                  reinterpret_cast<const float4 *>(smem + L::kOffU + r * L::kKvStride + (2 * sl + hh) * L::kSlot);
#pragma unroll
              for (int i = 0; i < DH / 4; ++i) {
                const float4 v = ap[i];
                av[hh * DH + 4 * i] = v.x, av[hh * DH + 4 * i + 1] = v.y;
                av[hh * DH + 4 * i + 2] = v.z, av[hh * DH + 4 * i + 3] = v.w;
              }
            }
          } else {
            tc_fence_after();  // the tasks' TMEM stores of other warps are ordered by the barrier above
            tmem_ld<XS>(tl + sl * XS, av);
            tmem_wait_ld();
            // heads whose task ran off this quadrant: A from their slots
            const uint32_t qg = qtab[qd];
            if (qg != 0xFFu) {
#pragma unroll
              for (int hh = 0; hh < 2; ++hh) {
                const uint32_t qs = qtab[4 + qg * 8 + 2 * sl + hh];
                if (qs != 0xFFu) {
#pragma unroll
                  for (int f = 0; f < DH / 4; ++f) {
                    const float4 v = ld_shared_f4(qslot_piece(qs, lane, f));
                    av[hh * DH + 4 * f] = v.x, av[hh * DH + 4 * f + 1] = v.y;
                    av[hh * DH + 4 * f + 2] = v.z, av[hh * DH + 4 * f + 3] = v.w;
                  }
                }
              }
            }
          }
          if constexpr (LIN == 1) {
            store_bf16<XS>(aop, r, sl * XS, D, av);
          } else {
            float amax = 0.0f;
#pragma unroll
            for (int j = 0; j < XS; ++j) amax = fmaxf(amax, fabsf(av[j]));
            float a = word_alpha(row_max(amax));
            a = (a > p.alpha_floor) ? a : p.alpha_floor;
            alpha_in = a;
            const float rr = __fdiv_rn(127.0f, a);
            float qv[XS];
            codes<XS>(av, rr, qv);
            store_codes<XS>(aop, r, sl * XS, D, qv);
            if (cap) capture_q(l, 1, qv, sl * XS, XS, alpha_in);
          }
        } else if constexpr (!STAGED) {
          cluster_arrive(bar_kvr);
          cluster_wait(bar_kvr, kvr_ph);

          // ---------------- S5: HPSA (Sec. 4.2)
          // the A of each head goes over the head's Q in TMEM (this thread's lane; that Q has no
          // other reader), so that the second head's attention runs with the registers of one;
          // d = 32 (d_h = 4, below the TMEM store width) keeps both in registers
          constexpr bool kStashA = DH >= 8;
          float A[kStashA ? 1 : 2][DH];
          float amax = 0.0f;
  #pragma unroll
          for (int hh = 0; hh < 2; ++hh) {
            const int e = sl + 4 * hh;
            float *Ah = A[kStashA ? 0 : hh];
            float qa[DH], bq[DH];
            ldg_vec<DH>(lp + LP::bqkv(D) + e * DH, bq);
            tmem_ld<DH>(tl + e * DH, qa);
            tmem_wait_ld();
            if (cap) capture_acc(l, 0, qa, e * DH, DH);
            float q[DH];
  #pragma unroll
            for (int i = 0; i < DH; ++i) q[i] = __fadd_rn(__fmul_rn(qa[i], fq), bq[i]);
  #pragma unroll
            for (int i = 0; i < DH; ++i) Ah[i] = 0.0f;
            {
              const int mk = (e < p.h_first) ? 0 : 1;
              constexpr int U = (DH >= 16) ? 2 : 4;
              // this thread's score cache: its own TMEM lane, kRowCache columns per column slice
              const uint32_t tcache = tl + L::kRowCacheCol + static_cast<uint32_t>(sl) * kRowCache;
              const uint32_t info = row_cw ? __ldg(p.mask_info[mk] + t) : 0u;
              if (p.C == 1)
                hpsa_head<DH, U, L::kKvStride, false>(q, info, row_cw, p.mask_list[mk], smem + L::kOffU, s_kvcl,
                                                      g * Tp, e * (8 * DH), p.att_scale, tcache, Ah);
              else
                hpsa_head<DH, U, L::kKvStride, true>(q, info, row_cw, p.mask_list[mk], smem + L::kOffU, s_kvcl,
                                                     g * Tp, e * (8 * DH), p.att_scale, tcache, Ah);
            }
  #pragma unroll
            for (int i = 0; i < DH; ++i) amax = fmaxf(amax, fabsf(Ah[i]));
            if constexpr (kStashA) tmem_st<DH>(tl + e * DH, Ah);
          }
          if constexpr (kStashA) tmem_wait_st();
          // A of head sl + 4 hh, from TMEM or registers
          auto head_a = [&](int hh, float *out) {
            if constexpr (kStashA) {
              tmem_ld<DH>(tl + (sl + 4 * hh) * DH, out);
              tmem_wait_ld();
            } else {
#pragma unroll
              for (int i = 0; i < DH; ++i) out[i] = A[hh][i];
            }
          };
          // Quant(A) -> O operand
          if constexpr (LIN == 1) {
#pragma unroll
            for (int hh = 0; hh < 2; ++hh) {
              float ah[DH];
              head_a(hh, ah);
              store_bf16<DH>(aop, r, (sl + 4 * hh) * DH, D, ah);
            }
          } else {
            float a = word_alpha(row_max(amax));
            a = (a > p.alpha_floor) ? a : p.alpha_floor;
            alpha_in = a;
            const float rr = __fdiv_rn(127.0f, a);
  #pragma unroll
            for (int hh = 0; hh < 2; ++hh) {
              const int e = sl + 4 * hh;
              float ah[DH], qv[DH];
              head_a(hh, ah);
              codes<DH>(ah, rr, qv);
              store_codes<DH>(aop, r, e * DH, D, qv);
              if (cap) capture_q(l, 1, qv, e * DH, DH, alpha_in);
            }
          }
        } else {
          // ---------------- S5: HPSA (Sec. 4.2), per-row lists over per-head staged rows (d = 128).
          // Every CTA of the cluster has left the K and V rows of its token rows in the cluster's
          // scratch in global memory (L2).  Head by head, one bulk copy brings the K rows of the
          // head for every row of the group into a K buffer and another the V rows into a V buffer;
          // two sets of buffers (region U and the operand tile, idle here) let the next head's rows
          // arrive while this head computes.  The row's 4 threads share the head: each takes 4 keys of every 16-key block for the scores
          // and their exponentials (the row's TMEM lane, columns from kSc), and then folds every
          // key, in ascending order, into 4 of the 16 features of num.  The arithmetic is the
          // canonical one, key for key and feature for feature.
          // this CTA's K and V rows, from region U to the cluster's scratch in global memory: 16 bulk
          // copies (one per head and kind, 8 KB each) by thread 0, complete before the cluster
          // learns that they are there
          fence_proxy_async_smem();  // this thread's K / V stores, before the bulk copies read them
          named_bar_sync(5, kEpiThreads);
          if (tid == 0 && !*s_abort) {
            const int R = p.C * kRows;
            for (int ek = 0; ek < 2 * kHeads; ++ek)
              bulk_s2g(p.kv_scratch + (static_cast<size_t>(cluster_id) * 2 * kHeads + ek) * R * DH +
                           static_cast<size_t>(crank) * kRows * DH,
                       kvl + static_cast<uint32_t>(ek) * kRows * 64u, kRows * 64u);
            bulk_commit_group();
            bulk_wait_group_0();
            fence_proxy_async_global();
          }
          cluster_arrive(bar_kvr);
          cluster_wait(bar_kvr, kvr_ph);
          static_assert(L::kOffU == 0 && L::kOffAop == L::kRegionU &&
                            L::kRegionU + L::kAopBytes >= 4u * kStagedMaxRows * 64u,
                        "two sets of K and V buffers span region U and the operand tile");
          constexpr uint32_t kSc = 128;  // the dead K and V accumulator columns [128, 384)
          // row rho of the group: 64 bytes at rho * 64, 16-byte piece f at f ^ ((rho >> 1) & 3)
          const int nrows = p.G * Tp;  // <= 640 (checked at create)
          const int rowbase = g * Tp;
          const uint32_t fetch_bytes = static_cast<uint32_t>(nrows) * 64u;
          // two sets of K and V buffers in region U (its K and V went to the scratch: idle here) and
          // the operand tile, [K0 | V0 | K1 | V1]: head e uses set e & 1 and the next-but-one head is
          // fetched after head e, so each head needs one CTA barrier
          const float *kvs = p.kv_scratch + static_cast<size_t>(cluster_id) * kHeads * 2 * (p.C * kRows) * DH;
          auto buf_of = [&](int e, int kind) -> uint32_t {
            return sb + L::kOffU + (static_cast<uint32_t>(e & 1) * 2u + kind) * fetch_bytes;
          };
          auto bar_of = [&](int e, int kind) -> uint32_t { return (kind ? bar_sv : bar_sk) + ((e & 1) ? 16u : 0u); };
          // phase parity of head e's barrier: one completion per two heads, 4 a block
          auto par_of = [&](int e) -> uint32_t { return static_cast<uint32_t>((e >> 1) & 1); };
          // thread 0: the bulk copy of head e's K (kind 0) or V (kind 1) rows (nothing once a wait
          // gave up, so that the teardown knows every copy in flight)
          auto fetch = [&](int e, int kind) {
            if (*s_abort) return;
            const uint32_t bar = bar_of(e, kind);
            mbar_arrive_expect_tx(bar, fetch_bytes);
            bulk_g2s(buf_of(e, kind), kvs + (static_cast<size_t>(e) * 2 + kind) * (p.C * kRows) * DH, fetch_bytes,
                     bar);
            ++s_issued[6 + kind + ((e & 1) ? 2 : 0)];
          };
          if (tid == 0) fetch(0, 0), fetch(0, 1), fetch(1, 0), fetch(1, 1);
          auto dot16 = [&](const float *q, const float4 *kk) -> float {
            float2 d2 = make_float2(0.0f, 0.0f);
#pragma unroll
            for (int i = 0; i < DH / 4; ++i) {
              d2 = fma2(make_float2(q[4 * i], q[4 * i + 1]), make_float2(kk[i].x, kk[i].y), d2);
              d2 = fma2(make_float2(q[4 * i + 2], q[4 * i + 3]), make_float2(kk[i].z, kk[i].w), d2);
            }
            return __fadd_rn(d2.x, d2.y);
          };
          for (int e = 0; e < kHeads; ++e) {
            // each barrier completes 4 times a block: an even number
            const uint32_t ph = par_of(e);
            const uint32_t kbuf = buf_of(e, 0), vbuf = buf_of(e, 1);
            const int mk = (e < p.h_first) ? 0 : 1;
            const uint32_t info = row_cw ? __ldg(p.mask_info[mk] + t) : 0u;
            const int cnt = static_cast<int>(info & 2047u);
            const uint4 *lst = p.mask_list[mk] + (info >> 11);
            const int nmax = __reduce_max_sync(0xffffffffu, cnt);  // the same for the 4 warps of the quadrant
            float q[DH];
            {
              float qa[DH], bq[DH];
              ldg_vec<DH>(lp + LP::bqkv(D) + e * DH, bq);
              tmem_ld<DH>(tl + e * DH, qa);
              tmem_wait_ld();
              if (cap && sl == (e & 3)) capture_acc(l, 0, qa, e * DH, DH);
#pragma unroll
              for (int i = 0; i < DH; ++i) q[i] = __fadd_rn(__fmul_rn(qa[i], fq), bq[i]);
            }
            wait_bar_warp(ctl, bar_of(e, 0), ph, false);  // this head's K rows have landed
            // pass 1: sigma of keys [b + 4 sl, b + 4 sl + 4) of every 16-key block b, and their maximum
            float mx = -INFINITY;
            for (int b = 0; b < nmax; b += 16) {
              const int k0 = b + 4 * sl;
              if (k0 < nmax) {
                const uint4 w = (k0 < cnt) ? __ldg(lst + (k0 >> 3)) : make_uint4(0u, 0u, 0u, 0u);
                const uint32_t lo = (k0 & 4) ? w.z : w.x, hi = (k0 & 4) ? w.w : w.y;
                const int idx[4] = {static_cast<int>(lo & 0xFFFFu), static_cast<int>(lo >> 16),
                                    static_cast<int>(hi & 0xFFFFu), static_cast<int>(hi >> 16)};
                float sg[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                  const int rho = rowbase + idx[i];  // a key past the row's count reads a valid row (offset 0)
                  const uint32_t rb = kbuf + static_cast<uint32_t>(rho) * 64u;
                  float4 kk[DH / 4];
#pragma unroll
                  for (int f = 0; f < DH / 4; ++f)
                    kk[f] = ld_shared_f4(rb + static_cast<uint32_t>((f ^ ((rho >> 1) & 3)) << 4));
                  sg[i] = __fmul_rn(dot16(q, kk), p.att_scale);
                  if (k0 + i < cnt) mx = fmaxf(mx, sg[i]);
                }
                tmem_st4(tl + kSc + k0, sg[0], sg[1], sg[2], sg[3]);
              }
            }
            tmem_wait_st();
            tc_fence_before();
            mx = row_max(mx);
            tc_fence_after();
            // pass 2: p = 2^(sigma - m) of the same keys, written over their scores
            for (int b = 0; b < nmax; b += 16) {
              const int k0 = b + 4 * sl;
              if (k0 < nmax) {
                float sg[4];
                tmem_ld<4>(tl + kSc + k0, sg);
                tmem_wait_ld();
                const float2 p01 = exp2_series2(add2(make_float2(sg[0], sg[1]), make_float2(-mx, -mx)));
                const float2 p23 = exp2_series2(add2(make_float2(sg[2], sg[3]), make_float2(-mx, -mx)));
                tmem_st4(tl + kSc + k0, p01.x, p01.y, p23.x, p23.y);
              }
            }
            tmem_wait_st();
            tc_fence_before();
            named_bar_sync(qbar, 128);
            tc_fence_after();
            wait_bar_warp(ctl, bar_of(e, 1), ph, false);  // this head's V rows have landed
            // l = sum p and num = sum p v over the row's keys in ascending order, features [4 sl, 4 sl + 4)
            float lsum = 0.0f, num[4] = {0.0f, 0.0f, 0.0f, 0.0f};
            for (int b = 0; b < nmax; b += 16) {
              float pb[16];
              tmem_ld<16>(tl + kSc + b, pb);
              tmem_wait_ld();
              const uint4 w0 = (b < cnt) ? __ldg(lst + (b >> 3)) : make_uint4(0u, 0u, 0u, 0u);
              const uint4 w1 = (b + 8 < cnt) ? __ldg(lst + (b >> 3) + 1) : make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
              for (int kk = 0; kk < 16; ++kk) {
                if (b + kk < cnt) {
                  const int rho = rowbase + idx_at(kk < 8 ? w0 : w1, kk & 7);
                  const float4 vv = ld_shared_f4(vbuf + static_cast<uint32_t>(rho) * 64u +
                                                 static_cast<uint32_t>((sl ^ ((rho >> 1) & 3)) << 4));
                  lsum = __fadd_rn(lsum, pb[kk]);
                  num[0] = __fmaf_rn(pb[kk], vv.x, num[0]);
                  num[1] = __fmaf_rn(pb[kk], vv.y, num[1]);
                  num[2] = __fmaf_rn(pb[kk], vv.z, num[2]);
                  num[3] = __fmaf_rn(pb[kk], vv.w, num[3]);
                }
              }
            }
            {
              const float inv = __fdiv_rn(1.0f, lsum);
              float a4[4];
#pragma unroll
              for (int f = 0; f < 4; ++f) a4[f] = row_cw ? __fmul_rn(num[f], inv) : 0.0f;
              // A of (row, head e), features [4 sl, 4 sl + 4), over the head's Q (read by all 4 threads
              // before the barriers above)
              tmem_st4(tl + e * DH + 4 * sl, a4[0], a4[1], a4[2], a4[3]);
            }
            tmem_wait_st();
            tc_fence_before();
            // the row's four threads (the quadrant's warps) are past this head's reads of the
            // score columns, which the next head's pass 1 rewrites; after the last head every
            // attention output in TMEM is ordered before Quant(A)
            if (e == kHeads - 1) named_bar_sync(5, kEpiThreads);
            else named_bar_sync(qbar, 128);
            tc_fence_after();
            if (e + 2 < kHeads) {
              // this warp is past its reads of this head's buffers; the last warp of the CTA to get
              // here fetches the next-but-one head's K and V into them (no quadrant waits for the
              // slowest one between heads; a warp that runs ahead waits for those rows to land)
              if (lane == 0) {
                __threadfence_block();
                if (atomicAdd(s_headdone + (e & 1), 1u) == static_cast<uint32_t>(kEpiWarps - 1)) {
                  s_headdone[e & 1] = 0u;
                  __threadfence_block();
                  fence_proxy_async_smem();
                  fetch(e + 2, 0), fetch(e + 2, 1);
                }
              }
              __syncwarp();
            }
          }
          // Quant(A) -> O operand: columns [sl XS, sl XS + XS) = heads 2 sl and 2 sl + 1, from TMEM
          float av[XS];
          tmem_ld<XS>(tl + sl * XS, av);
          tmem_wait_ld();
          if constexpr (LIN == 1) {
            store_bf16<XS>(aop, r, sl * XS, D, av);
          } else {
            float amax = 0.0f;
#pragma unroll
            for (int j = 0; j < XS; ++j) amax = fmaxf(amax, fabsf(av[j]));
            float a = word_alpha(row_max(amax));
            a = (a > p.alpha_floor) ? a : p.alpha_floor;
            alpha_in = a;
            const float rr = __fdiv_rn(127.0f, a);
            float qv[XS];
            codes<XS>(av, rr, qv);
            store_codes<XS>(aop, r, sl * XS, D, qv);
            if (cap) capture_q(l, 1, qv, sl * XS, XS, alpha_in);
          }
        }
        // this CTA no longer reads any K/V of this block (arrived before the O GEMM is issued: the
        // d = 128 schedule stages FFN1's weights over the K/V region once every CTA has arrived)
        if constexpr (ATT == 0) cluster_arrive(bar_kvf);
        signal_op(1, l, gi);
        // staged mode: every fetch from the cluster's K/V scratch of this block has landed (the
        // last head's barrier); a thread of warp 1, which next waits for the O accumulators, tells
        // the cluster, off warp 0's path to the O GEMM
        if constexpr (STAGED) kvf_signal(32);

        // ---------------- S6: O projection + residual + LayerNorm (Sec. 5, Post-LN)
        {
          const float fo = dq_factor(sw + 3);
          float ac[XS], bb[XS];
          if constexpr (kEarlyBias) ldg_vec<XS>(lp + LP::bo(D) + sl * XS, bb);
          wait_acc();
          tmem_ld<XS>(tl + sl * XS, ac);
          tmem_ld<XS>(tl + 3 * D + sl * XS, x);
          tmem_wait_ld();
          if (cap) capture_acc(l, 1, ac, sl * XS, XS);
          if constexpr (!kEarlyBias) ldg_vec<XS>(lp + LP::bo(D) + sl * XS, bb);
          residual_ln(ac, fo, bb, lp + LP::ln1g(D) + sl * XS, lp + LP::ln1b(D) + sl * XS);
        }
        {
          const float rr = quant_x_to_aop();
          if (cap) {
            float qv[XS];
            codes<XS>(x, rr, qv);
            capture_q(l, 2, qv, sl * XS, XS, alpha_in);
          }
        }
        signal_op(2, l, gi);

        // ---------------- S7: FFN1 + ReLU (Sec. 4 item 4) or GELU, Quant(u) -> FFN2 operand
        {
          const float f1 = dq_factor(sw + 4);
          constexpr int NCH = D / 32;
          // accumulator column of this thread's chunk ch of 32 hidden units (units sl D + 32 ch +
          // [0, 32)).  d = 128 (ffn1_unit_of_column): chunks 0 and 1 in [64 sl, 64 sl + 64), done
          // with FFN1's first N-tile pair, chunks 2 and 3 in [256 + 64 sl, 256 + 64 sl + 64).
          auto acc_col = [&](int ch) -> int {
            if constexpr (D == 128) return ch < 2 ? 64 * sl + 32 * ch : 256 + 64 * sl + 32 * (ch - 2);
            else return sl * D + 32 * ch;
          };
          // before chunk ch.  d = 128: chunks 0 and 1 wait for the first half of FFN1's MMAs, 2 and 3
          // for all of them (the block's third accumulator phase); then warp 0 stages FFN2's
          // weights into region U, whose last readers, FFN1's MMAs, are complete
          auto wait_chunk = [&](int ch) {
            if constexpr (D == 128) {
              static_assert(16 * S + 48 + 64 == 160, "bar_fin + 64 is the issuer's bar_acc_lo");
              if (ch == 0 || ch == 2) {
                if (ch == 0) wait_bar_warp(ctl, bar_fin + 64, (blk_base + static_cast<uint32_t>(l)) & 1u, false);
                else wait_bar_warp(ctl, bar_acc, 0, false);
                tc_fence_after();
                if (ch == 2 && warp == 0) issuer.stage_ffn2(p.wstream + static_cast<size_t>(l) * p.layer_bytes);
              }
            } else {
              if (ch == 0) wait_acc();
            }
          };
          // ACT 0 = ReLU, 1 = GELU.  u = act(acc f1 + b1) in 32-column chunks of this thread's D
          // hidden units.  AAP: u is stored over its own accumulators in TMEM (this thread's lane
          // and columns) between the row maximum and the codes, which leaves the registers to the
          // rest of the kernel.  Full-precision linears: one pass, u rounded to bf16.
          auto hidden = [&](int ch, float *u, bool capture) {
            const int c0 = sl * D + 32 * ch;
            float ac[32], bb[32];
            tmem_ld<32>(tl + acc_col(ch), ac);
            tmem_wait_ld();
            if (capture) capture_acc(l, 2, ac, c0, 32);
            ldg_vec<32>(lp + LP::b1(D) + c0, bb);
            dequant<32>(ac, f1, bb, u);
#pragma unroll
            for (int j = 0; j < 32; ++j) u[j] = ACT == 0 ? (u[j] > 0.0f ? u[j] : 0.0f) : gelu_as(u[j]);
          };
          // d = 128: FFN2's operand goes to TMEM, the 32 values of chunk ch packed two to a column
          // into the 16 columns [64 sl + 16 ch, 64 sl + 16 ch + 16) of this thread's lane (hidden
          // unit h at column h / 2, the even one in the low half).  Those columns belong to chunks
          // 0 and 1, and the chunk that held them was read before (chunk order 0, 1, 2, 3).
          auto put_operand = [&](int ch, const uint32_t *w) {
            tmem_st_u32<16>(tl + 64 * sl + 16 * ch, w);
          };
          if constexpr (LIN == 1) {
            // peers have finished reading this CTA's K/V: the shared region may now take u
            if constexpr (!TASKS) cluster_wait(bar_kvf, kvf_ph);
#pragma unroll
            for (int ch = 0; ch < NCH; ++ch) {
              wait_chunk(ch);
              float u[32];
              hidden(ch, u, cap);
              if constexpr (D == 128) {
                uint32_t w[16];
#pragma unroll
                for (int i = 0; i < 16; ++i) w[i] = pack_bf16x2_rn(u[2 * i], u[2 * i + 1]);
                put_operand(ch, w);
              } else {
                store_bf16<32>(uqt, r, sl * D + 32 * ch, 4 * D, u);
              }
            }
            if constexpr (D == 128) tmem_wait_st();
          } else {
            float umax = 0.0f;
#pragma unroll
            for (int ch = 0; ch < NCH; ++ch) {
              wait_chunk(ch);
              float u[32];
              hidden(ch, u, cap);
#pragma unroll
              for (int j = 0; j < 32; ++j) umax = fmaxf(umax, fabsf(u[j]));
              tmem_st<32>(tl + acc_col(ch), u);
            }
            tmem_wait_st();
            float a = word_alpha(row_max(umax));
            a = (a > p.alpha_floor) ? a : p.alpha_floor;
            alpha_in = a;
            const float rr = __fdiv_rn(127.0f, a);
            // peers have finished reading this CTA's K/V: the shared region may now take u codes
            // (d <= 64; at d = 128 the staged attention's scratch is free for the next block's K/V)
            if constexpr (!TASKS) cluster_wait(bar_kvf, kvf_ph);
#pragma unroll
            for (int ch = 0; ch < NCH; ++ch) {
              const int c0 = sl * D + 32 * ch;
              float u[32];
              tmem_ld<32>(tl + acc_col(ch), u);
              tmem_wait_ld();
              float qv[32];
              codes<32>(u, rr, qv);
              if constexpr (D == 128) {
                uint32_t w[16];
#pragma unroll
                for (int i = 0; i < 16; ++i) w[i] = pack_bf16x2(qv[2 * i], qv[2 * i + 1]);
                put_operand(ch, w);
              } else {
                store_codes<32>(uqt, r, c0, 4 * D, qv);
              }
              if (cap) capture_q(l, 3, qv, c0, 32, alpha_in);
            }
            if constexpr (D == 128) tmem_wait_st();
          }
        }
        signal_op(3, l, gi);

        // ---------------- S8: FFN2 + residual + LayerNorm
        {
          const float f2 = dq_factor(sw + 5);
          float ac[XS], bb[XS];
          if constexpr (kEarlyBias) ldg_vec<XS>(lp + LP::b2(D) + sl * XS, bb);
          wait_acc();
          // d = 128: FFN2's accumulators sit after its operand in TMEM, columns [256, 384)
          tmem_ld<XS>(tl + (D == 128 ? 256 : 0) + sl * XS, ac);
          tmem_wait_ld();
          if (cap) capture_acc(l, 3, ac, sl * XS, XS);
          if constexpr (!kEarlyBias) ldg_vec<XS>(lp + LP::b2(D) + sl * XS, bb);
          residual_ln(ac, f2, bb, lp + LP::ln2g(D) + sl * XS, lp + LP::ln2b(D) + sl * XS);
        }
        if (l + 1 < p.n_layers) {
          const float rr = quant_x_to_aop();
          if (cap) {
            float qv[XS];
            codes<XS>(x, rr, qv);
            capture_q(l + 1, 0, qv, sl * XS, XS, alpha_in);
          }
          signal_op(0, l + 1, gi);
        }
      }

      // ---------------- S9: output head (Sec. 3): z_t = x_t . w_{d->1} + b, eps = W_o^T z + b_o
      {
        float wv[XS];
        ldg_vec<XS>(p.w_d1 + sl * XS, wv);
#pragma unroll
        for (int j = 0; j < XS; ++j) wv[j] = __fmul_rn(x[j], wv[j]);
        const float z = __fadd_rn(row_sum(psum<XS>(wv)), p.b_d1);
        if (z_uses > 0) cluster_wait(bar_zf, zf_ph);
        ++z_uses;
        if (sl == 0) zbuf[r] = z;
      }
      cluster_arrive(bar_zr);
      cluster_wait(bar_zr, zr_ph);
      // ---------------- S10: decisions x_hat = y * eps, decoded-word syndrome
      {
        const int n_local = (p.G - static_cast<int>(crank) + p.C - 1) / p.C;  // groups g = crank + C*i
        // z of this CTA's words in token order, gathered once (from peers' rows too) into the
        // reduction area, which is idle until the next group (n_local T <= 1024 floats)
        float *ztok = red.buf;
        for (int it = tid; it < n_local * T; it += kEpiThreads) {
          const int li = it / T, tt = it - li * T;
          const int ru = (static_cast<int>(crank) + li * p.C) * Tp + __ldg(p.pos + tt);
          ztok[it] = *reinterpret_cast<const float *>(s_zgen[ru >> 7] + static_cast<uint32_t>(ru & 127) * 4u);
        }
        named_bar_sync(5, kEpiThreads);
        // one warp per 32 variables of a word, so that the decoded bits come out as bitmask words
        const int witems = n_local * W * 32;
        for (int it = tid; it < (witems + 31) / 32 * 32; it += kEpiThreads) {
          const int li = it / (W * 32), j = it - li * (W * 32);
          const int gg = static_cast<int>(crank) + li * p.C;
          const int64_t bb = gi * p.G + gg;
          const bool valid = it < witems && j < n && bb < p.B;
          bool bit = false;
          if (valid) {
            // eps_j = sum over t in token order of W_o[t][j] z_t (one FMA chain), loads ahead
            const float *zl = ztok + li * T;
            const float *wo = p.w_out + j;
            float acc = 0.0f;
            int tt = 0;
            for (; tt + 8 <= T; tt += 8) {
              float wv[8];
#pragma unroll
              for (int u = 0; u < 8; ++u) wv[u] = __ldg(wo + (tt + u) * n);
#pragma unroll
              for (int u = 0; u < 8; ++u) acc = __fmaf_rn(wv[u], zl[tt + u], acc);
            }
            for (; tt < T; ++tt) acc = __fmaf_rn(__ldg(wo + tt * n), zl[tt], acc);
            const float eps = __fadd_rn(acc, __ldg(p.b_out + j));
            bit = __fmul_rn(__ldg(p.y + bb * n + j), eps) < 0.0f;  // y was staged; re-read from L1/L2
            p.bits[bb * n + j] = bit ? 1 : 0;
            if (p.logits) p.logits[bb * n + j] = eps;
          }
          const uint32_t word = __ballot_sync(0xffffffffu, bit);
          if (lane == 0 && it < witems) bitw[it / 32] = word;
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
            for (int w = 0; w < W; ++w) par += __popc(__ldg(p.hbits + i * W + w) & bitw[li * W + w]);
            p.syn[bb * m + i] = static_cast<uint8_t>(par & 1u);
          }
        }
        cluster_arrive(bar_zf);  // this CTA no longer reads any z of this group; obits free
      }
      blk_base += static_cast<uint32_t>(p.n_layers);
    }
  }

  // ------------------------------------------------------------ teardown
  if (warp == 0) {
    // every MMA and every weight copy this CTA started must have landed before TMEM and the
    // shared memory go away
    __syncwarp();
    mma_commit_warp(bar_fin);
    if (lane == 0) {
      wait_bar_drain(ctl, bar_fin, 0);
      issuer.drain();
      if constexpr (STAGED)  // the staged attention's bulk copies of K and V rows (two buffer sets)
        for (int i = 0; i < 4; ++i)
          if (s_issued[6 + i] > 0)
            wait_bar_drain(ctl, ((i & 1) ? bar_sv : bar_sk) + (i >= 2 ? 16u : 0u), (s_issued[6 + i] - 1u) & 1u);
    }
    __syncwarp();
  }
  tc_fence_before();
  cluster_sync_all();
  if (warp == 0) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, L::kTmemCols);
  }
}

template <int D, int ATT, int ACT, int LIN>
cudaError_t prepare_decode_kernel(int cluster_ctas, uint32_t plan_bytes, int *max_active_clusters) {
  using L = SmemLayout<D, ATT == 1>;
  const uint32_t total = L::kTotal + plan_bytes;
  cudaError_t e = cudaFuncSetAttribute(aecct_decoder_kernel<D, ATT, ACT, LIN>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(total));
  if (e != cudaSuccess) return e;
  // ask for the smallest shared-memory carve-out that holds one CTA (1 KB of it is reserved by
  // the system): the rest of the 256 KB unified array stays L1 for spills and parameter loads
  int dev = 0, smem_sm = 0;
  if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
  if ((e = cudaDeviceGetAttribute(&smem_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, dev)) != cudaSuccess)
    return e;
  if (smem_sm > 0) {
    const int pct = static_cast<int>((100ll * (total + 1024) + smem_sm - 1) / smem_sm);
    e = cudaFuncSetAttribute(aecct_decoder_kernel<D, ATT, ACT, LIN>, cudaFuncAttributePreferredSharedMemoryCarveout,
                             pct > 100 ? 100 : pct);
    if (e != cudaSuccess) return e;
  }
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = cluster_ctas;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.gridDim = dim3(cluster_ctas, 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = total;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaOccupancyMaxActiveClusters(max_active_clusters, aecct_decoder_kernel<D, ATT, ACT, LIN>, &cfg);
}

template <int D, int ATT, int ACT, int LIN>
cudaError_t launch_decode(const DecodeParams &p, cudaStream_t stream) {
  using L = SmemLayout<D, ATT == 1>;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = p.C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.gridDim = dim3(p.n_clusters * p.C, 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = L::kTotal + p.plan_bytes;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, aecct_decoder_kernel<D, ATT, ACT, LIN>, p);
}

}  // namespace aecct
