// Fused <SpMM,GEMM> on CUDA cores (and <SpMMH,GEMM>, whose gathered row is
// the Hadamard product C(k,:) .* C2(k,:)) over light rows, and the dense
// GEMM of the unfused variant.
//
// Fused schedule (Sec. 4.2, Algorithm 1 applied to A = B.C.D): the shared
// outer loop is the row i; the producer builds T(i,:) = sum_j B(i,j) C(j,:)
// and the consumer multiplies it by D at once.  Here a CTA owns a tile of
// kTileRows consecutive rows: the producer writes the tile's T rows into
// shared memory (never to global memory), the consumer multiplies the
// tile by D and writes A's rows once.  Rows with more than kLightMax
// nonzeros are left to the heavy-row path (spmm.cu).
#include "launch.h"
#include "tile.cuh"

namespace slnr {
namespace {

template <int K, bool H>
__global__ void __launch_bounds__(256) k_spmm_gemm_tiles(int nrows, const int32_t* __restrict__ pos,
                                                         const int32_t* __restrict__ crd,
                                                         const float* __restrict__ vals,
                                                         const float* __restrict__ C,
                                                         const float* __restrict__ C2,
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
        gather_acc<RL::VPL, H ? 2 : 4, H>(acc, crd, vals, p0, p1, C, K, col, C2);
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

// Row-fused variant for D of at most kRowsMaxD floats (staged whole in shared
// memory): lane groups build their rows' T in registers exactly as the row
// SpMM kernel does, then the warp multiplies each of its GPW rows by D in
// turn (T(k) broadcast by shuffles, OPL outputs per lane) and writes A's row
// once.  No tile barrier: gathers and products of different warps overlap.
constexpr int kRowsMaxD = 16384;

template <int K, int L, bool H>
__global__ void __launch_bounds__(256) k_spmm_gemm_rows(int nrows, const int32_t* __restrict__ pos,
                                                        const int32_t* __restrict__ crd,
                                                        const float* __restrict__ vals,
                                                        const float* __restrict__ C,
                                                        const float* __restrict__ C2,
                                                        const float* __restrict__ D, float* __restrict__ A) {
  using RL = RowLanes<K>;
  constexpr int VPL = RL::VPL, GS = RL::GS, GPW = RL::GPW;
  constexpr int OPL = L >= 32 ? L / 32 : 1, OL = L / OPL;  // outputs per lane, lanes with outputs
  static_assert(K * L <= kRowsMaxD && OPL <= 8, "D fits the shared stage; at most 8 outputs per lane");
  extern __shared__ float4 smem4[];
  const float* Ds = reinterpret_cast<const float*>(smem4);
  for (int i = threadIdx.x; i < K * L / 4; i += blockDim.x) smem4[i] = __ldg(reinterpret_cast<const float4*>(D) + i);
  __syncthreads();
  const int lane = threadIdx.x & 31, grp = lane / GS, col = (lane % GS) * VPL;
  const int64_t gwarp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t r0 = gwarp * GPW; r0 < nrows; r0 += nwarps * GPW) {
    // producer: group g builds T(r0 + g, :) in registers
    const int64_t r = r0 + grp;
    float t[VPL];
    zero_vec(t);
    int light = 0;
    if (r < nrows) {
      const int p0 = pos[r], p1 = pos[r + 1];
      if (p1 - p0 <= kLightMax) {
        gather_acc<VPL, H ? 2 : 4, H>(t, crd, vals, p0, p1, C, K, col, C2);
        light = 1;
      }
    }
    // consumer: A(r0 + q, :) = T(r0 + q, :) . D for each light row q of the warp
#pragma unroll 1
    for (int q = 0; q < GPW; ++q) {
      const int64_t rq = r0 + q;
      if (rq >= nrows) break;                                        // warp-uniform
      if (!__shfl_sync(0xffffffffu, light, q * GS)) continue;        // heavy: the combine writes it
      float a[OPL];
#pragma unroll
      for (int o = 0; o < OPL; ++o) a[o] = 0.f;
#pragma unroll 1
      for (int c = 0; c < GS; ++c) {  // lane q*GS + c of the warp holds T(c*VPL .. c*VPL + VPL)
#pragma unroll
        for (int e = 0; e < VPL; ++e) {
          const float tv = __shfl_sync(0xffffffffu, t[e], q * GS + c);
          const float* drow = Ds + (c * VPL + e) * L + lane * OPL;
          if (lane < OL) {
#pragma unroll
            for (int o = 0; o < OPL; ++o) a[o] = fmaf(tv, drow[o], a[o]);
          }
        }
      }
      if (lane < OL) {
        float* dst = A + rq * L + lane * OPL;
        if constexpr (OPL % 4 == 0) {
#pragma unroll
          for (int o = 0; o < OPL; o += 4) *reinterpret_cast<float4*>(dst + o) = make_float4(a[o], a[o + 1], a[o + 2], a[o + 3]);
        } else {
#pragma unroll
          for (int o = 0; o < OPL; ++o) dst[o] = a[o];
        }
      }
    }
  }
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

}  // namespace

cudaError_t launch_spmm_gemm_tiles(int K, int L, const CsrView& B, const float* C, const float* D,
                                   float* A, int use_tf32, cudaStream_t s, const float* C2) {
  (void)use_tf32;
  if (B.nrows <= 0) return cudaSuccess;
  // The row kernel reads all of D from shared memory once per row; the tile
  // kernel reuses each staged D element across 32 rows.  Measured on the
  // 2^20-row R-MAT graph, the row kernel is faster for L <= 64 and for
  // K L < 4096 (and D must fit its stage).
  if (K * L <= kRowsMaxD && (L <= 64 || K * L < 4096)) {  // row-fused kernel, D staged whole
    const size_t smem = sizeof(float) * (size_t)K * (size_t)L;
    SLNR_WIDTH_SWITCH(K, KC, {
      SLNR_WIDTH_SWITCH(L, LC, {
        if constexpr (KC * LC <= kRowsMaxD) {
          constexpr int GPW = RowLanes<KC>::GPW;
          int64_t ctas = ceil_div(ceil_div(B.nrows, GPW), 8);
          const int64_t cap = (int64_t)device_sm_count() * 16;
          if (ctas > cap) ctas = cap;
          if (C2 == nullptr) {
            cudaError_t e = set_smem(k_spmm_gemm_rows<KC, LC, false>, smem);
            if (e != cudaSuccess) return e;
            k_spmm_gemm_rows<KC, LC, false><<<SLNR_COUNTED((unsigned)ctas), 256, smem, s>>>(B.nrows, B.pos, B.crd, B.vals, C,
                                                                               nullptr, D, A);
          } else {
            cudaError_t e = set_smem(k_spmm_gemm_rows<KC, LC, true>, smem);
            if (e != cudaSuccess) return e;
            k_spmm_gemm_rows<KC, LC, true><<<SLNR_COUNTED((unsigned)ctas), 256, smem, s>>>(B.nrows, B.pos, B.crd, B.vals, C, C2,
                                                                              D, A);
          }
        }
      });
    });
    return cudaGetLastError();
  }
  const int64_t grid = ceil_div(B.nrows, kTileRows);
  const size_t smem = tile_smem_bytes(K, L);
  SLNR_WIDTH_SWITCH(K, KC, {
    if (C2 == nullptr) {
      cudaError_t e = set_smem(k_spmm_gemm_tiles<KC, false>, smem);
      if (e != cudaSuccess) return e;
      k_spmm_gemm_tiles<KC, false><<<SLNR_COUNTED((unsigned)grid), 256, smem, s>>>(B.nrows, B.pos, B.crd, B.vals, C, nullptr, D,
                                                                     L, A);
    } else {
      cudaError_t e = set_smem(k_spmm_gemm_tiles<KC, true>, smem);
      if (e != cudaSuccess) return e;
      k_spmm_gemm_tiles<KC, true><<<SLNR_COUNTED((unsigned)grid), 256, smem, s>>>(B.nrows, B.pos, B.crd, B.vals, C, C2, D, L,
                                                                    A);
    }
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
    k_dense_gemm<KC><<<SLNR_COUNTED((unsigned)grid), 256, smem, s>>>(M, T, D, L, A);
  });
  return cudaGetLastError();
}

}  // namespace slnr
