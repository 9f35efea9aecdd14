// Peaks of this GPU, measured by the library's own kernels: the FP32 FFMA
// rate of the CUDA cores and the TF32 rate of the tcgen05 tensor cores (the
// two kinds of arithmetic the consumer contractions run on), and the rate of
// whole-row gathers from a table (the producers' loads).  They are the
// compute and gather denominators of the roofline the benchmark reports.
#include <algorithm>

#include "launch.h"
#include "tcgen05.cuh"

namespace slnr {
namespace {

constexpr int kFfmaThreads = 256;
constexpr int kFfmaChains = 8;  // independent FMA chains per thread

// Each thread runs kFfmaChains independent chains of `iters` dependent FMAs
// (2 flops each).  The values stay finite; `sink` is written only if a value
// happens to equal a given number, so the arithmetic cannot be dropped.
__global__ void __launch_bounds__(kFfmaThreads) k_peak_ffma(int64_t iters, float seed, float* sink) {
  float a[kFfmaChains];
#pragma unroll
  for (int c = 0; c < kFfmaChains; ++c) a[c] = seed + 0.001f * (float)(threadIdx.x + c);
  const float m = 0.9999f, k = 1e-4f;
  for (int64_t i = 0; i < iters; ++i)
#pragma unroll
    for (int c = 0; c < kFfmaChains; ++c) a[c] = fmaf(a[c], m, k);
  float s = 0.f;
#pragma unroll
  for (int c = 0; c < kFfmaChains; ++c) s += a[c];
  if (sink != nullptr && s == 1234.5f) sink[0] = s;
}

// One CTA per SM: thread 0 issues `passes` x 4 tcgen05.mma (kind::tf32,
// M = 128, N = 256, K = 8; 2 * 128 * 256 * 8 flops each) on operands in
// shared memory, accumulating into 256 tensor-memory columns, then commits
// and waits (bounded) for completion.
constexpr int kMmaM = 128, kMmaN = 256;

// Set by k_peak_tf32 if its wait for the MMAs gave up.
__device__ int g_peak_flag;

__global__ void __launch_bounds__(128, 1) k_peak_tf32(int64_t passes) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ uint64_t done;
  __shared__ uint32_t tmem_base;
  uint8_t* sA = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sB = sA + kMmaM * 128;  // one 128-byte swizzle block of A (128 rows x 32 tf32)
  const int warp = threadIdx.x >> 5;
  for (int i = threadIdx.x; i < (kMmaM + kMmaN) * 32; i += blockDim.x)
    reinterpret_cast<uint32_t*>(sA)[i] = tc::to_tf32(0.25f + 0.001f * (float)(i % 97));
  if (warp == 0) {
    tc::tmem_alloc(&tmem_base, kMmaN);
    tc::tmem_relinquish();
  }
  if (threadIdx.x == 0) {
    tc::mbar_init(&done, 1);
    tc::fence_mbar_init();
  }
  tc::fence_proxy_async_smem();
  tc::tc_fence_before_sync();
  __syncthreads();
  tc::tc_fence_after_sync();
  const uint32_t tmem = tmem_base;
  if (threadIdx.x == 0) {
    constexpr uint32_t idesc = tc::idesc_tf32(kMmaM, kMmaN);
    const uint32_t a = tc::smem_u32(sA), b = tc::smem_u32(sB);
    for (int64_t p = 0; p < passes; ++p)
#pragma unroll
      for (int ks = 0; ks < 4; ++ks)
        tc::mma_tf32(tmem, tc::desc_k_sw128(a + 32 * ks), tc::desc_k_sw128(b + 32 * ks), idesc, (p | ks) != 0);
    tc::mma_commit(&done);
    // bounded wait; on a timeout a second bounded wait drains the MMAs
    // before the tensor memory is released
    for (int attempt = 0; attempt < 2; ++attempt) {
      const long long t0 = clock64();
      bool ok = true;
      while (!tc::mbar_try_wait(&done, 0))
        if (clock64() - t0 > kWaitCycles) {
          ok = false;
          break;
        }
      if (ok) break;
      atomicOr(&g_peak_flag, kErrTimeout);
    }
  }
  tc::tc_fence_before_sync();
  __syncthreads();
  tc::tc_fence_after_sync();
  if (warp == 0) tc::tmem_dealloc(tmem, kMmaN);
}

constexpr int kGatherThreads = 256;
constexpr int kGatherBatch = 8;  // rows in flight per lane group

// Row gathers, as the producers of the fused kernels issue them: a lane group
// of q = width / 4 lanes reads a whole row of a rows x width fp32 table (one
// float4 per lane) at a pseudo-random row id, kGatherBatch rows in flight,
// and keeps a running sum.  Row ids come from a per-group linear
// congruential sequence (the Numerical Recipes constants) mapped to
// [0, rows) by a multiply-shift.  `sink` is written only if the sum equals
// a given number, so the loads cannot be dropped.
__global__ void __launch_bounds__(kGatherThreads) k_peak_gather(const float4* __restrict__ table, uint32_t rows,
                                                                int q, int iters, float* sink) {
  const int lane = threadIdx.x & 31, g = lane / q, c = lane % q;
  const uint32_t group = (blockIdx.x * (kGatherThreads / 32) + (threadIdx.x >> 5)) * (32 / q) + g;
  uint32_t x = group * 0x9E3779B9u + 0x7F4A7C15u;
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  for (int i = 0; i < iters; ++i) {
    float4 v[kGatherBatch];
#pragma unroll
    for (int u = 0; u < kGatherBatch; ++u) {
      x = x * 1664525u + 1013904223u;
      const uint32_t r = (uint32_t)(((uint64_t)(x ^ (x >> 16)) * rows) >> 32);
      v[u] = __ldg(table + (int64_t)r * q + c);
    }
#pragma unroll
    for (int u = 0; u < kGatherBatch; ++u) {
      acc.x += v[u].x;
      acc.y += v[u].y;
      acc.z += v[u].z;
      acc.w += v[u].w;
    }
  }
  if (sink != nullptr && acc.x + acc.y + acc.z + acc.w == 1234.5f) sink[0] = acc.x;
}

template <typename F>
cudaError_t timed(cudaStream_t s, float* ms, F launch) {
  cudaEvent_t a, b;
  cudaError_t e = cudaEventCreate(&a);
  if (e != cudaSuccess) return e;
  if ((e = cudaEventCreate(&b)) != cudaSuccess) {
    cudaEventDestroy(a);
    return e;
  }
  if ((e = launch()) == cudaSuccess && (e = cudaEventRecord(a, s)) == cudaSuccess &&
      (e = launch()) == cudaSuccess && (e = cudaEventRecord(b, s)) == cudaSuccess &&
      (e = cudaEventSynchronize(b)) == cudaSuccess)
    e = cudaEventElapsedTime(ms, a, b);
  cudaEventDestroy(a);
  cudaEventDestroy(b);
  return e;
}

}  // namespace

cudaError_t peak_ffma(cudaStream_t s, double* tflops) {
  const int64_t iters = 1 << 16;
  const int grid = device_sm_count() * 8;
  float ms = 0.f;
  cudaError_t e = timed(s, &ms, [&] {
    k_peak_ffma<<<grid, kFfmaThreads, 0, s>>>(iters, 1.0f, nullptr);
    return cudaGetLastError();
  });
  if (e != cudaSuccess) return e;
  *tflops = 2.0 * kFfmaChains * (double)iters * grid * kFfmaThreads / (ms * 1e-3) / 1e12;
  return cudaSuccess;
}

cudaError_t peak_tf32(cudaStream_t s, double* tflops) {
  const int64_t passes = 1 << 13;
  const int grid = device_sm_count();
  // the operands take 49 KB; ask for 120 KB so that one CTA runs per SM
  const size_t smem = (size_t)120 * 1024;
  cudaError_t e = cudaFuncSetAttribute(k_peak_tf32, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  const int zero = 0;
  if ((e = cudaMemcpyToSymbolAsync(g_peak_flag, &zero, sizeof(int), 0, cudaMemcpyHostToDevice, s)) != cudaSuccess)
    return e;
  float ms = 0.f;
  e = timed(s, &ms, [&] {
    k_peak_tf32<<<grid, 128, smem, s>>>(passes);
    return cudaGetLastError();
  });
  if (e != cudaSuccess) return e;
  int flag = 0;
  if ((e = cudaMemcpyFromSymbol(&flag, g_peak_flag, sizeof(int))) != cudaSuccess) return e;
  if (flag != 0) return cudaErrorLaunchTimeout;
  *tflops = 2.0 * kMmaM * kMmaN * 8 * 4 * (double)passes * grid / (ms * 1e-3) / 1e12;
  return cudaSuccess;
}

cudaError_t peak_gather(const float* table, int64_t rows, int width, cudaStream_t s, double* gbs) {
  const int q = width / 4;
  const int grid = device_sm_count() * (2048 / kGatherThreads);
  const int64_t groups = (int64_t)grid * (kGatherThreads / 32) * (32 / q);
  const int64_t row_bytes = (int64_t)width * 4;
  // about 4 GB of gathered rows per launch
  const int iters = (int)std::max<int64_t>(1, ((int64_t)4 << 30) / (groups * kGatherBatch * row_bytes));
  float ms = 0.f;
  cudaError_t e = timed(s, &ms, [&] {
    k_peak_gather<<<grid, kGatherThreads, 0, s>>>(reinterpret_cast<const float4*>(table), (uint32_t)rows, q, iters,
                                                  nullptr);
    return cudaGetLastError();
  });
  if (e != cudaSuccess) return e;
  *gbs = (double)groups * iters * kGatherBatch * row_bytes / (ms * 1e-3) / 1e9;
  return cudaSuccess;
}

}  // namespace slnr
