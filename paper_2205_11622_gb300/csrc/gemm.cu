// Fused <SpMM,GEMM> over light rows, and the dense GEMM of the unfused
// variant.
//
// Fused schedule (Sec. 4.2, Algorithm 1 applied to A = B.C.D): the shared
// outer loop is the row i; the producer builds T(i,:) = sum_j B(i,j) C(j,:)
// and the consumer multiplies it by D at once.  Here a CTA owns a tile of
// kTileRows consecutive rows: the producer writes the tile's T rows into
// shared memory (never to global memory), the consumer multiplies the
// tile by D and writes A's rows once.  Rows with more than kLightMax
// nonzeros are left to the heavy-row path (spmm.cu).
#include "launch.h"

namespace slnr {
namespace {

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

template <int K>
__global__ void __launch_bounds__(256) k_spmm_gemm_tiles(int nrows, const int32_t* __restrict__ pos,
                                                         const int32_t* __restrict__ crd,
                                                         const float* __restrict__ vals,
                                                         const float* __restrict__ C,
                                                         const float* __restrict__ D, int L,
                                                         float* __restrict__ A) {
  using RL = RowLanes<K>;
  extern __shared__ float4 smem4[];
  float* T = reinterpret_cast<float*>(smem4);
  float* Ds = T + kTileRows * K;
  __shared__ int keep[kTileRows];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int grp = lane / RL::GS, col = (lane % RL::GS) * RL::VPL;
  const int64_t r0 = (int64_t)blockIdx.x * kTileRows;
  // producer: T rows of the tile, on chip
  for (int rr = warp * RL::GPW + grp; rr < kTileRows; rr += 8 * RL::GPW) {
    const int64_t r = r0 + rr;
    float acc[RL::VPL];
    zero_vec(acc);
    int ok = 0;
    if (r < nrows) {
      const int p0 = pos[r], p1 = pos[r + 1];
      if (p1 - p0 <= kLightMax) {
        gather_acc<RL::VPL>(acc, crd, vals, p0, p1, C, K, col);
        ok = 1;
      }
    }
    st_vec(T + rr * K + col, acc);
    if (col == 0) keep[rr] = ok;
  }
  __syncthreads();
  // consumer: A rows = T . D
  tile_times_d<K>(T, D, L, Ds, A, r0, nrows, keep);
}

template <int K>
__global__ void __launch_bounds__(256) k_dense_gemm(int64_t M, const float* __restrict__ Tg,
                                                    const float* __restrict__ D, int L,
                                                    float* __restrict__ A) {
  extern __shared__ float4 smem4[];
  float* T = reinterpret_cast<float*>(smem4);
  float* Ds = T + kTileRows * K;
  const int64_t r0 = (int64_t)blockIdx.x * kTileRows;
  constexpr int N4 = kTileRows * K / 4;
  for (int i = threadIdx.x; i < N4; i += blockDim.x) {
    const int rr = i / (K / 4);
    float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
    if (r0 + rr < M) v = __ldg(reinterpret_cast<const float4*>(Tg + r0 * K) + i);
    smem4[i] = v;
  }
  __syncthreads();
  tile_times_d<K>(T, D, L, Ds, A, r0, M, nullptr);
}

// Opt in to more than the default 48 KB of dynamic shared memory (the
// kernels also hold a little static shared memory).
template <typename Kern>
cudaError_t set_smem(Kern k, size_t bytes) {
  if (bytes <= 40 * 1024) return cudaSuccess;
  return cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
}

}  // namespace

cudaError_t launch_spmm_gemm_tiles(int K, int L, const CsrView& B, const float* C, const float* D,
                                   float* A, int use_tf32, cudaStream_t s) {
  (void)use_tf32;
  if (B.nrows <= 0) return cudaSuccess;
  const int64_t grid = ceil_div(B.nrows, kTileRows);
  const size_t smem = sizeof(float) * ((size_t)kTileRows * K + (size_t)d_chunk_rows(K, L) * L);
  SLNR_WIDTH_SWITCH(K, KC, {
    cudaError_t e = set_smem(k_spmm_gemm_tiles<KC>, smem);
    if (e != cudaSuccess) return e;
    k_spmm_gemm_tiles<KC><<<(unsigned)grid, 256, smem, s>>>(B.nrows, B.pos, B.crd, B.vals, C, D, L, A);
  });
  return cudaGetLastError();
}

cudaError_t launch_dense_gemm(int64_t M, int K, int L, const float* T, const float* D, float* A,
                              int use_tf32, cudaStream_t s) {
  (void)use_tf32;
  if (M <= 0) return cudaSuccess;
  const int64_t grid = ceil_div(M, kTileRows);
  const size_t smem = sizeof(float) * ((size_t)kTileRows * K + (size_t)d_chunk_rows(K, L) * L);
  SLNR_WIDTH_SWITCH(K, KC, {
    cudaError_t e = set_smem(k_dense_gemm<KC>, smem);
    if (e != cudaSuccess) return e;
    k_dense_gemm<KC><<<(unsigned)grid, 256, smem, s>>>(M, T, D, L, A);
  });
  return cudaGetLastError();
}

}  // namespace slnr
