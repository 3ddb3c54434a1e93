// aap.cu -- the AAP weight quantiser of Sec. 4.1 (eq. Ternary) on the GPU, as the training forward
// applies it, and the expansion of 2-bit ternary weights into the decoder's bf16 tile stream.
//
// aap_ternarize_kernel: one CTA per weight tensor.
//   gamma = Percentile(|W|, 0.5): the median of |W| with linear interpolation between the two
//     middle order statistics (position 0.5 (len - 1)), the two order statistics found exactly by
//     a most-significant-digit radix select over the bit patterns of |W| (for non-negative
//     floats the bit patterns order like the values), the interpolation in double precision;
//   scale = gamma * delta (fp32), t = RoundClip(W / (scale + eps), -1, 1) with an IEEE fp32
//     division and round to nearest even;
//   t goes out in the 2-bit format of aecct_create (weight i at bits 2 (i % 4) of byte i / 4:
//     00 = 0, 01 = +1, 11 = -1), and optionally as the training forward's weight scale * t.
// unpack_weights_kernel: the 2-bit weights of aecct_create, expanded on the GPU into bf16 K-major
//   core-matrix chunks in WeightSchedule order (one 16-byte core-matrix row per thread).
#include <cuda_runtime.h>

#include <cstdint>

#include "aecct_internal.h"

namespace aecct {

namespace {

constexpr int kSelectThreads = 1024;

// the k-th smallest (0-based) of the keys |w_i| (bit patterns, sign cleared) of one tensor
__device__ uint32_t radix_select(const float *w, int64_t len, int64_t k, uint32_t *hist, uint32_t *sel) {
  uint32_t prefix = 0, mask = 0;
  for (int shift = 24; shift >= 0; shift -= 8) {
    for (int b = threadIdx.x; b < 256; b += blockDim.x) hist[b] = 0;
    __syncthreads();
    for (int64_t i = threadIdx.x; i < len; i += blockDim.x) {
      const uint32_t key = __float_as_uint(w[i]) & 0x7FFFFFFFu;
      if ((key & mask) == prefix) atomicAdd(&hist[(key >> shift) & 0xFFu], 1u);
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      uint64_t cum = 0;
      uint32_t b = 0;
      for (; b < 255; ++b) {
        if (cum + hist[b] > static_cast<uint64_t>(k)) break;
        cum += hist[b];
      }
      sel[0] = b;
      sel[1] = static_cast<uint32_t>(cum);
    }
    __syncthreads();
    const uint32_t b = sel[0];
    k -= sel[1];
    prefix |= b << shift;
    mask |= 0xFFu << shift;
    __syncthreads();
  }
  return prefix;
}

struct TernarizeArgs {
  int n;
  int64_t off[kTernarizeMaxTensors];  // first element of tensor j in w (and of its codes * 4)
  int64_t len[kTernarizeMaxTensors];
  float delta[kTernarizeMaxTensors];
};

__global__ void __launch_bounds__(kSelectThreads) aap_ternarize_kernel(const float *__restrict__ w, const TernarizeArgs a,
                                                                       float eps, uint8_t *packed, float *scale,
                                                                       float *wq) {
  __shared__ uint32_t hist[256];
  __shared__ uint32_t sel[2];
  __shared__ float s_den, s_sc;
  const int j = blockIdx.x;
  const float *wt = w + a.off[j];
  const int64_t len = a.len[j];
  // Percentile(|W|, 0.5): position 0.5 (len - 1) between the order statistics lo and lo + 1
  const double pos = 0.5 * static_cast<double>(len - 1);
  const int64_t lo = static_cast<int64_t>(floor(pos));
  const int64_t hi = lo + 1 < len ? lo + 1 : lo;
  const double frac = pos - static_cast<double>(lo);
  const uint32_t klo = radix_select(wt, len, lo, hist, sel);
  const uint32_t khi = hi == lo ? klo : radix_select(wt, len, hi, hist, sel);
  if (threadIdx.x == 0) {
    const double alo = static_cast<double>(__uint_as_float(klo)), ahi = static_cast<double>(__uint_as_float(khi));
    const float gamma = static_cast<float>(alo + frac * (ahi - alo));
    const float sc = __fmul_rn(gamma, a.delta[j]);
    scale[j] = sc;
    s_sc = sc;
    s_den = __fadd_rn(sc, eps);
  }
  __syncthreads();
  const float den = s_den, sc = s_sc;
  uint8_t *pk = packed + a.off[j] / 4;
  for (int64_t q = threadIdx.x; q < len / 4; q += blockDim.x) {
    uint32_t byte = 0;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float v = rintf(__fdiv_rn(wt[4 * q + i], den));
      // RoundClip to the integers {-1, 0, +1} (a rounded -0 is the integer 0)
      const float t = v >= 1.0f ? 1.0f : (v <= -1.0f ? -1.0f : 0.0f);
      byte |= (t > 0.0f ? 1u : (t < 0.0f ? 3u : 0u)) << (2 * i);
      if (wq) wq[a.off[j] + 4 * q + i] = __fmul_rn(sc, t);
    }
    pk[q] = static_cast<uint8_t>(byte);
  }
}

struct UnpackArgs {
  int D, n_chunks;
  uint32_t layer_bytes;
  ChunkDesc chunk[32];
};

// one thread per (layer, chunk, row, 8-column group): 8 ternary codes (2 bytes of the packed row)
// -> one 16-byte core-matrix row of bf16
__global__ void unpack_weights_kernel(const uint8_t *__restrict__ packed, int n_layers, const UnpackArgs a,
                                      uint8_t *wstream) {
  const int D = a.D, F = 4 * D;
  const size_t per_layer_packed = 3u * static_cast<size_t>(D) * D;  // 12 D^2 weights / 4
  int64_t item = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  // items per layer: sum over chunks of nrows * kcols / 8
  int64_t per_layer = 0;
  for (int c = 0; c < a.n_chunks; ++c) per_layer += static_cast<int64_t>(a.chunk[c].nrows) * a.chunk[c].kcols / 8;
  if (item >= per_layer * n_layers) return;
  const int l = static_cast<int>(item / per_layer);
  item -= static_cast<int64_t>(l) * per_layer;
  int c = 0;
  for (; c < a.n_chunks; ++c) {
    const int64_t n = static_cast<int64_t>(a.chunk[c].nrows) * a.chunk[c].kcols / 8;
    if (item < n) break;
    item -= n;
  }
  const ChunkDesc ch = a.chunk[c];
  const int rr = static_cast<int>(item / (ch.kcols / 8)), cg = static_cast<int>(item % (ch.kcols / 8));
  const int n = ch.n0 + rr, k = ch.k0 + 8 * cg;
  // the ABI tensor and row of GEMM row n: QKV rows [0, D) W_q, [D, 2D) W_k, [2D, 3D) W_v; O W_o;
  // FFN1 W_1 [F][D] (output column n holds hidden unit ffn1_unit_of_column(D, n)); FFN2 W_2 [D][F]
  size_t toff;
  int row, din;
  if (ch.gemm == 0) toff = static_cast<size_t>(n / D) * D * D / 4, row = n % D, din = D;
  else if (ch.gemm == 1) toff = 3u * static_cast<size_t>(D) * D / 4, row = n, din = D;
  else if (ch.gemm == 2) toff = static_cast<size_t>(D) * D, row = ffn1_unit_of_column(D, n), din = D;
  else toff = static_cast<size_t>(D) * D + static_cast<size_t>(F) * D / 4, row = n, din = F;
  const uint8_t *src = packed + per_layer_packed * l + toff + static_cast<size_t>(row) * (din / 4) + k / 4;
  const uint32_t bits = static_cast<uint32_t>(src[0]) | (static_cast<uint32_t>(src[1]) << 8);
  uint32_t h[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    uint32_t pair = 0;
#pragma unroll
    for (int s = 0; s < 2; ++s) {
      const uint32_t code = (bits >> (2 * (2 * i + s))) & 3u;
      const uint32_t bf = code == 1u ? 0x3F80u : (code == 3u ? 0xBF80u : 0u);  // +1, -1, 0 in bf16
      pair |= bf << (16 * s);
    }
    h[i] = pair;
  }
  uint8_t *dst = wstream + static_cast<size_t>(l) * a.layer_bytes + ch.off + core_off(rr, 8 * cg, ch.kcols);
  *reinterpret_cast<uint4 *>(dst) = make_uint4(h[0], h[1], h[2], h[3]);
}

}  // namespace

cudaError_t launch_aap_ternarize(const float *w, int n, const int64_t *len, const float *delta, float eps,
                                 uint8_t *packed, float *scale, float *wq, cudaStream_t stream) {
  int64_t off = 0;
  for (int j0 = 0; j0 < n; j0 += kTernarizeMaxTensors) {
    TernarizeArgs a = {};
    a.n = n - j0 < kTernarizeMaxTensors ? n - j0 : kTernarizeMaxTensors;
    int64_t first = off;
    for (int j = 0; j < a.n; ++j) {
      a.off[j] = off - first;
      a.len[j] = len[j0 + j];
      a.delta[j] = delta[j0 + j];
      off += len[j0 + j];
    }
    aap_ternarize_kernel<<<a.n, kSelectThreads, 0, stream>>>(w + first, a, eps, packed + first / 4, scale + j0,
                                                              wq ? wq + first : nullptr);
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

cudaError_t launch_unpack_weights(const uint8_t *packed, int n_layers, int D, const ChunkDesc *chunks, int n_chunks,
                                  uint32_t layer_bytes, uint8_t *wstream, cudaStream_t stream) {
  UnpackArgs a = {};
  a.D = D, a.n_chunks = n_chunks, a.layer_bytes = layer_bytes;
  int64_t per_layer = 0;
  for (int c = 0; c < n_chunks; ++c) {
    a.chunk[c] = chunks[c];
    per_layer += static_cast<int64_t>(chunks[c].nrows) * chunks[c].kcols / 8;
  }
  const int64_t items = per_layer * n_layers;
  const int threads = 256;
  unpack_weights_kernel<<<static_cast<unsigned>((items + threads - 1) / threads), threads, 0, stream>>>(packed, n_layers,
                                                                                                        a, wstream);
  return cudaGetLastError();
}

}  // namespace aecct
