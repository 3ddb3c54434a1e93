// selftest.cu -- diagnostics kernels of libaecct (no counterpart in the paper).
//
// selftest_mma_kernel: stages A [128][K] and B [N][K] in the same K-major no-swizzle core-matrix
// layout the decoder uses, runs tcgen05.mma (kind::f16, bf16 operands, fp32 accumulators in
// TMEM) and reads the accumulators back with tcgen05.ld.  It checks the descriptor encodings
// and the TMEM lane/column mapping on a single tile.
//
// selftest_timeout_kernel: one warp waits on an mbarrier that nothing completes, with a bounded
// wait; it reports that the wait gave up.  Nothing asynchronous is in flight while it waits.
#include <cuda_runtime.h>

#include "aecct_internal.h"
#include "sm103_ptx.cuh"

namespace aecct {

constexpr int kSelftestMaxK = 128;
constexpr int kSelftestMaxN = 256;

__global__ void __launch_bounds__(128, 1)
    selftest_mma_kernel(const int8_t *__restrict__ a, const int8_t *__restrict__ b, int K, int N, uint32_t tcols,
                        float *__restrict__ out, int *__restrict__ status, long long limit) {
  extern __shared__ __align__(1024) uint8_t smem[];
  const uint32_t sb = smem_u32(smem);
  const uint32_t a_tile = sb;
  const uint32_t b_tile = sb + 128u * kSelftestMaxK * 2u;
  const uint32_t bar = b_tile + kSelftestMaxN * kSelftestMaxK * 2u;
  uint32_t *s_tmem = reinterpret_cast<uint32_t *>(smem + (bar - sb) + 8);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  // stage the operands as bf16 (exact for int8 values)
  for (int i = tid; i < 128 * K; i += blockDim.x) {
    const int r = i / K, c = i - r * K;
    const __nv_bfloat16 v = __float2bfloat16_rn(static_cast<float>(a[i]));
    *reinterpret_cast<__nv_bfloat16 *>(smem + core_off(r, c, K)) = v;
  }
  for (int i = tid; i < N * K; i += blockDim.x) {
    const int r = i / K, c = i - r * K;
    const __nv_bfloat16 v = __float2bfloat16_rn(static_cast<float>(b[i]));
    *reinterpret_cast<__nv_bfloat16 *>(smem + (b_tile - sb) + core_off(r, c, K)) = v;
  }
  if (tid == 0) {
    mbar_init(bar, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0) {
    tmem_alloc(smem_u32(s_tmem), tcols);
    tmem_relinquish();
  }
  fence_proxy_async_smem();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *s_tmem;

  if (tid == 0) {
    const uint32_t idesc = make_idesc_bf16(128, N);
    const uint32_t sbo = (K / 8u) * 128u;
    for (int ks = 0; ks < K / 16; ++ks) {
      const uint64_t ad = make_sdesc(a_tile + ks * 256u, 128u, sbo);
      const uint64_t bd = make_sdesc(b_tile + ks * 256u, 128u, sbo);
      mma_bf16(tmem, ad, bd, idesc, ks > 0 ? 1u : 0u);
    }
    mma_commit(bar);
  }
  // every thread waits (bounded) for the accumulators
  bool ok = false;
  {
    const long long t0 = clock64();
    while (!(ok = mbar_try_wait(bar, 0))) {
      if (clock64() - t0 > limit) break;
    }
  }
  if (!ok && tid == 0) atomicExch(status, 1);
  tc_fence_after();
  const uint32_t tl = tmem + (static_cast<uint32_t>(32 * warp) << 16);
  const int r = 32 * warp + lane;
  for (int c0 = 0; c0 < N; c0 += 16) {
    float v[16];
    tmem_ld16(tl + c0, v);
    tmem_wait_ld();
#pragma unroll
    for (int j = 0; j < 16; ++j) out[r * N + c0 + j] = v[j];
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, tcols);
  }
}

__global__ void selftest_timeout_kernel(long long limit, int *status) {
  __shared__ __align__(8) uint64_t bar_storage;
  const uint32_t bar = smem_u32(&bar_storage);
  if (threadIdx.x == 0) mbar_init(bar, 1);
  __syncwarp();
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  __syncwarp();
  bool done = false;
  const long long t0 = clock64();
  while (!(done = mbar_try_wait(bar, 0))) {
    if (clock64() - t0 > limit) break;
  }
  if (threadIdx.x == 0) *status = done ? 0 : 1;
}

// fp32 fused multiply-add rate: every thread runs 8 independent FMA chains (scalar fma.rn.f32,
// or paired fma.rn.f32x2 with two FMAs per instruction) for `iters` steps; the values stay in
// [0, 1] (x <- x * 0.5 + 0.25 converges to 0.5), and a comparison nothing satisfies keeps the
// chains from being removed
template <bool PAIRED>
__global__ void __launch_bounds__(512) selftest_fma_kernel(int iters, float *sink) {
  const float s = 0.5f, c = 0.25f;
  if constexpr (PAIRED) {
    uint64_t a[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const float v = 0.001f * static_cast<float>(threadIdx.x + i);
      asm("mov.b64 %0, {%1, %2};" : "=l"(a[i]) : "f"(v), "f"(-v));
    }
    uint64_t sc, cc;
    asm("mov.b64 %0, {%1, %1};" : "=l"(sc) : "f"(s));
    asm("mov.b64 %0, {%1, %1};" : "=l"(cc) : "f"(c));
    for (int it = 0; it < iters; ++it) {
#pragma unroll
      for (int i = 0; i < 8; ++i) asm volatile("fma.rn.f32x2 %0, %0, %1, %2;" : "+l"(a[i]) : "l"(sc), "l"(cc));
    }
    float t = 0.0f;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      float lo, hi;
      asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(a[i]));
      t += lo + hi;
    }
    if (t == -1.0f) sink[blockIdx.x * blockDim.x + threadIdx.x] = t;
  } else {
    float a[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) a[i] = 0.001f * static_cast<float>(threadIdx.x + i);
    for (int it = 0; it < iters; ++it) {
#pragma unroll
      for (int i = 0; i < 8; ++i) asm volatile("fma.rn.f32 %0, %0, %1, %2;" : "+f"(a[i]) : "f"(s), "f"(c));
    }
    float t = 0.0f;
#pragma unroll
    for (int i = 0; i < 8; ++i) t += a[i];
    if (t == -1.0f) sink[blockIdx.x * blockDim.x + threadIdx.x] = t;
  }
}

cudaError_t run_selftest_fma_rate(bool paired, double *fma_per_s) {
  int dev = 0, sms = 0;
  cudaError_t e;
  if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
  if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
  const int blocks = 4 * sms, threads = 512, iters = 1 << 15;
  float *sink = nullptr;
  cudaEvent_t t0 = nullptr, t1 = nullptr;
  float best_ms = 0.0f;
  if ((e = cudaMalloc(&sink, sizeof(float) * blocks * threads)) != cudaSuccess) return e;
  if ((e = cudaEventCreate(&t0)) != cudaSuccess || (e = cudaEventCreate(&t1)) != cudaSuccess) goto done;
  for (int rep = 0; rep < 4; ++rep) {  // the first launch warms up
    if ((e = cudaEventRecord(t0)) != cudaSuccess) goto done;
    if (paired) selftest_fma_kernel<true><<<blocks, threads>>>(iters, sink);
    else selftest_fma_kernel<false><<<blocks, threads>>>(iters, sink);
    if ((e = cudaGetLastError()) != cudaSuccess) goto done;
    if ((e = cudaEventRecord(t1)) != cudaSuccess || (e = cudaEventSynchronize(t1)) != cudaSuccess) goto done;
    float ms = 0.0f;
    if ((e = cudaEventElapsedTime(&ms, t0, t1)) != cudaSuccess) goto done;
    if (rep > 0 && (best_ms == 0.0f || ms < best_ms)) best_ms = ms;
  }
  *fma_per_s = static_cast<double>(blocks) * threads * iters * 8.0 * (paired ? 2.0 : 1.0) / (best_ms * 1e-3);
done:
  if (t0) cudaEventDestroy(t0);
  if (t1) cudaEventDestroy(t1);
  cudaFree(sink);
  return e;
}

cudaError_t run_selftest_mma(const int8_t *a_host, const int8_t *b_host, int K, int N, float *out_host) {
  int8_t *da = nullptr, *db = nullptr;
  float *dout = nullptr;
  int *dst = nullptr;
  cudaError_t e;
  const size_t smem_bytes = 128u * kSelftestMaxK * 2u + kSelftestMaxN * kSelftestMaxK * 2u + 64u;
  uint32_t tcols = 32;
  while (tcols < static_cast<uint32_t>(N)) tcols <<= 1;
  int status = 0;
  if ((e = cudaMalloc(&da, 128 * K)) != cudaSuccess) goto done;
  if ((e = cudaMalloc(&db, N * K)) != cudaSuccess) goto done;
  if ((e = cudaMalloc(&dout, sizeof(float) * 128 * N)) != cudaSuccess) goto done;
  if ((e = cudaMalloc(&dst, sizeof(int))) != cudaSuccess) goto done;
  if ((e = cudaMemcpy(da, a_host, 128 * K, cudaMemcpyHostToDevice)) != cudaSuccess) goto done;
  if ((e = cudaMemcpy(db, b_host, N * K, cudaMemcpyHostToDevice)) != cudaSuccess) goto done;
  if ((e = cudaMemset(dst, 0, sizeof(int))) != cudaSuccess) goto done;
  if ((e = cudaFuncSetAttribute(selftest_mma_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                static_cast<int>(smem_bytes))) != cudaSuccess)
    goto done;
  selftest_mma_kernel<<<1, 128, smem_bytes>>>(da, db, K, N, tcols, dout, dst, 1LL << 31);
  if ((e = cudaGetLastError()) != cudaSuccess) goto done;
  if ((e = cudaDeviceSynchronize()) != cudaSuccess) goto done;
  if ((e = cudaMemcpy(out_host, dout, sizeof(float) * 128 * N, cudaMemcpyDeviceToHost)) != cudaSuccess) goto done;
  if ((e = cudaMemcpy(&status, dst, sizeof(int), cudaMemcpyDeviceToHost)) != cudaSuccess) goto done;
  if (status) e = cudaErrorTimeout;
done:
  cudaFree(da);
  cudaFree(db);
  cudaFree(dout);
  cudaFree(dst);
  return e;
}

cudaError_t run_selftest_timeout(long long limit_cycles, int *status_host) {
  int *dst = nullptr;
  cudaError_t e = cudaMalloc(&dst, sizeof(int));
  if (e != cudaSuccess) return e;
  int init = -1;
  if ((e = cudaMemcpy(dst, &init, sizeof(int), cudaMemcpyHostToDevice)) == cudaSuccess) {
    selftest_timeout_kernel<<<1, 32>>>(limit_cycles, dst);
    if ((e = cudaGetLastError()) == cudaSuccess && (e = cudaDeviceSynchronize()) == cudaSuccess)
      e = cudaMemcpy(status_host, dst, sizeof(int), cudaMemcpyDeviceToHost);
  }
  cudaFree(dst);
  return e;
}

}  // namespace aecct
