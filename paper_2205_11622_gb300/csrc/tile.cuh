// The FFMA consumer of the row-tile kernels: a CTA's tile of kTileRows
// temporary rows, held in shared memory, times a small dense matrix.
#pragma once

#include "common.cuh"

namespace slnr {

constexpr int kTileRows = 32;

// Rows of D staged in shared memory per step (KC x L <= 4096 floats).
__host__ __device__ constexpr int d_chunk_rows(int K, int L) { return K < 4096 / L ? K : 4096 / L; }

// A[r0 + rr, :] = T[rr, :] . D for rr in [0, kTileRows), rows < nrows with keep[rr]
// (keep == nullptr keeps all).  T: kTileRows x K in shared memory; D: K x L
// in global memory, staged through Ds (d_chunk_rows(K, L) x L floats).
// Every output is a k-ordered fp32 FMA chain.
template <int K>
__device__ __forceinline__ void tile_times_d(const float* T, const float* __restrict__ D, int L, float* Ds,
                                             float* __restrict__ A, int64_t r0, int64_t nrows,
                                             const int* keep) {
  const int ncg = L / 4;
  int rpt = (kTileRows * ncg) / 256;
  if (rpt < 1) rpt = 1;
  const int active = kTileRows * ncg / rpt;
  const int tid = threadIdx.x;
  const int cg = tid % ncg, rg = tid / ncg;
  const int KC = d_chunk_rows(K, L);
  float acc[8][4];
#pragma unroll
  for (int i = 0; i < 8; ++i) acc[i][0] = acc[i][1] = acc[i][2] = acc[i][3] = 0.f;
  for (int k0 = 0; k0 < K; k0 += KC) {
    for (int i = tid; i < KC * ncg; i += blockDim.x) {
      const int kk = i / ncg, c = i % ncg;
      reinterpret_cast<float4*>(Ds)[i] = __ldg(reinterpret_cast<const float4*>(D + (int64_t)(k0 + kk) * L) + c);
    }
    __syncthreads();
    if (tid < active) {
      for (int kk = 0; kk < KC; ++kk) {
        const float4 d = reinterpret_cast<const float4*>(Ds)[kk * ncg + cg];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          if (i < rpt) {
            const float t = T[(rg * rpt + i) * K + k0 + kk];
            acc[i][0] = fmaf(t, d.x, acc[i][0]);
            acc[i][1] = fmaf(t, d.y, acc[i][1]);
            acc[i][2] = fmaf(t, d.z, acc[i][2]);
            acc[i][3] = fmaf(t, d.w, acc[i][3]);
          }
        }
      }
    }
    __syncthreads();
  }
  if (tid < active) {
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      if (i < rpt) {
        const int rr = rg * rpt + i;
        const int64_t r = r0 + rr;
        if (r < nrows && (keep == nullptr || keep[rr]))
          reinterpret_cast<float4*>(A + r * L)[cg] = make_float4(acc[i][0], acc[i][1], acc[i][2], acc[i][3]);
      }
    }
  }
}

// Opt in to more than the default 48 KB of dynamic shared memory (the
// kernels also hold a little static shared memory).
template <typename Kern>
inline cudaError_t set_smem(Kern k, size_t bytes) {
  if (bytes <= 40 * 1024) return cudaSuccess;
  return cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
}

// Dynamic shared memory of a row-tile kernel: the T tile (kTileRows x K) and
// the staged rows of the consumer matrix (K x L).
inline size_t tile_smem_bytes(int K, int L) {
  return sizeof(float) * ((size_t)kTileRows * K + (size_t)d_chunk_rows(K, L) * L);
}

}  // namespace slnr
