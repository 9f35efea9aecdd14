// <SDDMM,SpMM>:  A(i,k) = sum_j B(i,j) * (sum_l C(i,l) D(j,l)) * E(j,k)
//
// Fused schedule (Fig. 2d; Sec. 4.2 finds the temporary to be a scalar):
// the shared loops are i and the stored j of row i; for each stored (i,j)
// the producer forms y = B(i,j) * <C(i,:), D(j,:)> and the consumer adds
// y * E(j,:) to A(i,:) at once.  A warp owns a row; its lane groups take
// successive nonzeros, C(i,:) stays in registers, the dot product is a group
// shuffle reduction, and the groups' A rows are summed at the end.  Heavy
// rows are split into chunks whose partial A rows are combined in a fixed
// order (spmm.cu, k_combine).
//
// Unfused schedule (Fig. 2a then Fig. 2b): Y(i,j) for every stored (i,j) is
// written to memory, then A = Y.E runs as an SpMM (spmm.cu).
#include "launch.h"
#include "tile.cuh"

#ifndef SLNR_SDDMM_MIN_CTAS
#define SLNR_SDDMM_MIN_CTAS 4  // resident 256-thread CTAs per SM the fused kernels are compiled for (64 registers)
#endif
constexpr int kRowsPerClaim = 4;  // rows a warp of the fused row kernel takes at a time
constexpr int kShortRow = 8;      // a claim whose rows all have at most this many nonzeros: a lane group per row

#ifndef SLNR_SDDMM_U
#define SLNR_SDDMM_U 2  // nonzeros in flight per lane group
#endif

namespace slnr {
namespace {


// Accumulates, for nonzeros p = p0 + grp, p0 + grp + GPW, ... < p1:
//   acc += vals[p] * <c, D(crd[p], :)> * E(crd[p], :)
// Every lane of the warp runs the same number of steps (shuffles stay
// converged); lanes past the end use zero weights and load nothing.
template <int WM, int U = SLNR_SDDMM_U>
__device__ __forceinline__ void sddmm_spmm_range(float (&acc)[RowLanes<WM>::VPL],
                                                 const float (&c)[RowLanes<WM>::VPL], int p0, int p1,
                                                 const int32_t* __restrict__ crd,
                                                 const float* __restrict__ vals,
                                                 const float* __restrict__ D, int L,
                                                 const float* __restrict__ E, int K, int grp, int col) {
  using RL = RowLanes<WM>;
  constexpr int VPL = RL::VPL;
  const int n = p1 - p0;
  for (int base = 0; base < n; base += RL::GPW * U) {
    int cc[U];
    float vv[U];
    bool ok[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int p = p0 + base + u * RL::GPW + grp;
      ok[u] = p < p1;
      cc[u] = ok[u] ? __ldg(crd + p) : 0;
      vv[u] = ok[u] ? __ldg(vals + p) : 0.f;
    }
    float d[U][VPL], e[U][VPL];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      if (ok[u] && col < L) ldg_vec_upto<VPL>(d[u], D + (int64_t)cc[u] * L + col, L - col); else zero_vec(d[u]);
      if (ok[u] && col < K) ldg_vec_upto<VPL>(e[u], E + (int64_t)cc[u] * K + col, K - col); else zero_vec(e[u]);
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      float dot = 0.f;
#pragma unroll
      for (int x = 0; x < VPL; ++x) dot = fmaf(c[x], d[u][x], dot);
      dot = group_sum<RL::GS>(dot);
      const float y = vv[u] * dot;
#pragma unroll
      for (int x = 0; x < VPL; ++x) acc[x] = fmaf(y, e[u][x], acc[x]);
    }
  }
}

// One launch for all of a call's work: warps take items from the header's
// counter, first the chunks of heavy rows (partial A rows into the
// workspace, summed later by k_combine), then blocks of kRowsPerClaim light
// rows (A rows written once).  Row lengths follow a power law, so the
// costly hub chunks start first and every warp stays busy until the counter
// runs out.
// A row of at most kShortRow nonzeros owned by one lane group: for each
// nonzero in order, acc += vals[p] <c, D(crd[p], :)> E(crd[p], :), U nonzeros
// in flight.  The trip count is the warp's longest row (maxlen, the same in
// every lane: the dot products' shuffles need the whole warp); shorter rows'
// slots are predicated off.
template <int WM, int U = SLNR_SDDMM_U>
__device__ __forceinline__ void short_row_range(float (&acc)[RowLanes<WM>::VPL],
                                                const float (&c)[RowLanes<WM>::VPL], int p0, int p1, int maxlen,
                                                const int32_t* __restrict__ crd, const float* __restrict__ vals,
                                                const float* __restrict__ D, int L, const float* __restrict__ E,
                                                int K, int col) {
  using RL = RowLanes<WM>;
  constexpr int VPL = RL::VPL;
  for (int it = 0; it < maxlen; it += U) {
    const int base = p0 + it;
    int cc[U];
    float vv[U];
    bool ok[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      ok[u] = base + u < p1;
      cc[u] = ok[u] ? __ldg(crd + base + u) : 0;
      vv[u] = ok[u] ? __ldg(vals + base + u) : 0.f;
    }
    float d[U][VPL], e[U][VPL];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      if (ok[u] && col < L) ldg_vec_upto<VPL>(d[u], D + (int64_t)cc[u] * L + col, L - col); else zero_vec(d[u]);
      if (ok[u] && col < K) ldg_vec_upto<VPL>(e[u], E + (int64_t)cc[u] * K + col, K - col); else zero_vec(e[u]);
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      float dot = 0.f;
#pragma unroll
      for (int x = 0; x < VPL; ++x) dot = fmaf(c[x], d[u][x], dot);
      dot = group_sum<RL::GS>(dot);
      const float y = vv[u] * dot;
#pragma unroll
      for (int x = 0; x < VPL; ++x) acc[x] = fmaf(y, e[u][x], acc[x]);
    }
  }
}

template <int WM>
__global__ void __launch_bounds__(256, SLNR_SDDMM_MIN_CTAS) k_sddmm_spmm_rows(WsHeader* hdr, int nrows,
                                                                              const int32_t* __restrict__ pos,
                                                                              const int32_t* __restrict__ crd,
                                                                              const float* __restrict__ vals,
                                                                              const float* __restrict__ C,
                                                                              const float* __restrict__ D, int L,
                                                                              const float* __restrict__ E, int K,
                                                                              float* __restrict__ A,
                                                                              const Chunk* __restrict__ chunks,
                                                                              int max_chunks,
                                                                              float* __restrict__ partial) {
  using RL = RowLanes<WM>;
  const int lane = threadIdx.x & 31, grp = lane / RL::GS, col = (lane % RL::GS) * RL::VPL;
  const int nch = min(hdr->n_chunks, max_chunks);
  for (;;) {
    int w = 0;
    if (lane == 0) w = atomicAdd(&hdr->next_row, 1);
    w = __shfl_sync(0xffffffffu, w, 0);
    if (w < nch) {  // a chunk of a heavy row
      const Chunk ch = chunks[w];
      float c[RL::VPL], acc[RL::VPL];
      if (col < L) ldg_vec_upto<RL::VPL>(c, C + (int64_t)ch.row * L + col, L - col); else zero_vec(c);
      zero_vec(acc);
      sddmm_spmm_range<WM>(acc, c, ch.p0, ch.p1, crd, vals, D, L, E, K, grp, col);
      cross_group_sum<RL::GS>(acc);
      if (grp == 0 && col < K) st_vec_upto(partial + (int64_t)ch.slot * K + col, acc, K - col);
      continue;
    }
    const int64_t r0 = (int64_t)(w - nch) * kRowsPerClaim;
    if (r0 >= nrows) break;
    const int64_t r1 = r0 + kRowsPerClaim < nrows ? r0 + kRowsPerClaim : nrows;
    // short rows: one row per lane group (no cross-group sum), nonzeros in order
    if constexpr (RL::GPW >= kRowsPerClaim) {
      const int64_t rg = r0 + grp;
      int gp0 = 0, gp1 = 0;
      if (grp < kRowsPerClaim && rg < r1) {
        gp0 = pos[rg];
        gp1 = pos[rg + 1];
      }
      const int maxlen = __reduce_max_sync(0xffffffffu, gp1 - gp0);
      if (maxlen <= kShortRow) {  // warp-uniform
        float c[RL::VPL], acc[RL::VPL];
        zero_vec(acc);
        if (gp1 > gp0 && col < L) ldg_vec_upto<RL::VPL>(c, C + rg * L + col, L - col); else zero_vec(c);
        short_row_range<WM>(acc, c, gp0, gp1, maxlen, crd, vals, D, L, E, K, col);
        if (grp < kRowsPerClaim && rg < r1 && col < K) st_vec_upto(A + rg * K + col, acc, K - col);
        continue;
      }
    }
    for (int64_t r = r0; r < r1; ++r) {
      const int p0 = pos[r], p1 = pos[r + 1];
      if (p1 - p0 > kLightMax) continue;  // warp-uniform: its chunks above
      float c[RL::VPL], acc[RL::VPL];
      if (col < L) ldg_vec_upto<RL::VPL>(c, C + r * L + col, L - col); else zero_vec(c);
      zero_vec(acc);
      sddmm_spmm_range<WM>(acc, c, p0, p1, crd, vals, D, L, E, K, grp, col);
      cross_group_sum<RL::GS>(acc);
      if (grp == 0 && col < K) st_vec_upto(A + r * K + col, acc, K - col);
    }
  }
}

template <int WM>
__global__ void __launch_bounds__(256, SLNR_SDDMM_MIN_CTAS) k_sddmm_spmm_chunks(const WsHeader* __restrict__ hdr,
                                                           const Chunk* __restrict__ chunks, int max_chunks,
                                                           const int32_t* __restrict__ crd,
                                                           const float* __restrict__ vals,
                                                           const float* __restrict__ C,
                                                           const float* __restrict__ D, int L,
                                                           const float* __restrict__ E, int K,
                                                           float* __restrict__ partial) {
  using RL = RowLanes<WM>;
  const int n = min(hdr->n_chunks, max_chunks);
  const int lane = threadIdx.x & 31, grp = lane / RL::GS, col = (lane % RL::GS) * RL::VPL;
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t w = warp; w < n; w += nwarps) {
    const Chunk ch = chunks[w];
    float c[RL::VPL], acc[RL::VPL];
    if (col < L) ldg_vec_upto<RL::VPL>(c, C + (int64_t)ch.row * L + col, L - col); else zero_vec(c);
    zero_vec(acc);
    sddmm_spmm_range<WM>(acc, c, ch.p0, ch.p1, crd, vals, D, L, E, K, grp, col);
    cross_group_sum<RL::GS>(acc);
    if (grp == 0 && col < K) st_vec_upto(partial + (int64_t)ch.slot * K + col, acc, K - col);
  }
}

// Fused <SDDMM,SpMM,GEMM> over light rows (Algorithm 1 applied twice): a CTA
// owns kTileRows consecutive rows; a warp builds a row's temporary
// T(i,:) = sum_j B(i,j) <C(i,:), D(j,:)> F(j,:) (scalar per nonzero, vector
// of width LW per row) into the shared-memory tile, then the tile is
// multiplied by W (LW x M) and A's rows are written once.  Rows with more than
// kLightMax nonzeros are left to the chunk kernel and k_combine (times W).
template <int WM, int LW>
__global__ void __launch_bounds__(256, SLNR_SDDMM_MIN_CTAS) k_sddmm_spmm_gemm_tiles(int nrows, const int32_t* __restrict__ pos,
                                                               const int32_t* __restrict__ crd,
                                                               const float* __restrict__ vals,
                                                               const float* __restrict__ C,
                                                               const float* __restrict__ D, int K,
                                                               const float* __restrict__ F,
                                                               const float* __restrict__ W, int M,
                                                               float* __restrict__ A) {
  using RL = RowLanes<WM>;
  extern __shared__ float4 smem4[];
  float* T = reinterpret_cast<float*>(smem4);
  float* Ws = T + kTileRows * LW;
  __shared__ int keep[kTileRows];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int grp = lane / RL::GS, col = (lane % RL::GS) * RL::VPL;
  const int64_t r0 = (int64_t)blockIdx.x * kTileRows;
  for (int rr = warp; rr < kTileRows; rr += 8) {
    const int64_t r = r0 + rr;
    float c[RL::VPL], acc[RL::VPL];
    zero_vec(acc);
    int ok = 0;
    if (r < nrows) {
      const int p0 = pos[r], p1 = pos[r + 1];
      if (p1 - p0 <= kLightMax) {  // warp-uniform
        if (col < K) ldg_vec_upto<RL::VPL>(c, C + r * K + col, K - col); else zero_vec(c);
        sddmm_spmm_range<WM>(acc, c, p0, p1, crd, vals, D, K, F, LW, grp, col);
        cross_group_sum<RL::GS>(acc);
        ok = 1;
      }
    }
    if (grp == 0 && col < LW) {
#pragma unroll
      for (int x = 0; x < RL::VPL; ++x)
        if (col + x < LW) T[rr * LW + col + x] = acc[x];
    }
    if (lane == 0) keep[rr] = ok;
  }
  __syncthreads();
  tile_times_d<LW>(T, W, M, Ws, A, r0, nrows, keep);
}

// Unfused producer: Y[p] = vals[p] * <C(i,:), D(crd[p],:)> for p in [p0, p1) of row i.
template <int W>
__device__ __forceinline__ void sddmm_range(const float (&c)[RowLanes<W>::VPL], int p0, int p1,
                                            const int32_t* __restrict__ crd, const float* __restrict__ vals,
                                            const float* __restrict__ D, float* __restrict__ Y, int grp,
                                            int col, int gl) {
  using RL = RowLanes<W>;
  const int n = p1 - p0;
  for (int base = 0; base < n; base += RL::GPW) {
    const int p = p0 + base + grp;
    const bool ok = p < p1;
    float d[RL::VPL];
    if (ok) ldg_vec<RL::VPL>(d, D + (int64_t)__ldg(crd + p) * W + col); else zero_vec(d);
    float dot = 0.f;
#pragma unroll
    for (int x = 0; x < RL::VPL; ++x) dot = fmaf(c[x], d[x], dot);
    dot = group_sum<RL::GS>(dot);
    if (ok && gl == 0) Y[p] = __ldg(vals + p) * dot;
  }
}

template <int W>
__global__ void __launch_bounds__(256) k_sddmm_rows(int nrows, const int32_t* __restrict__ pos,
                                                    const int32_t* __restrict__ crd,
                                                    const float* __restrict__ vals,
                                                    const float* __restrict__ C,
                                                    const float* __restrict__ D, float* __restrict__ Y) {
  using RL = RowLanes<W>;
  const int lane = threadIdx.x & 31, grp = lane / RL::GS, gl = lane % RL::GS, col = gl * RL::VPL;
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t r = warp; r < nrows; r += nwarps) {
    const int p0 = pos[r], p1 = pos[r + 1];
    if (p1 - p0 > kLightMax) continue;
    float c[RL::VPL];
    ldg_vec<RL::VPL>(c, C + r * W + col);
    sddmm_range<W>(c, p0, p1, crd, vals, D, Y, grp, col, gl);
  }
}

template <int W>
__global__ void __launch_bounds__(256) k_sddmm_chunks(const WsHeader* __restrict__ hdr,
                                                      const Chunk* __restrict__ chunks, int max_chunks,
                                                      const int32_t* __restrict__ crd,
                                                      const float* __restrict__ vals,
                                                      const float* __restrict__ C,
                                                      const float* __restrict__ D, float* __restrict__ Y) {
  using RL = RowLanes<W>;
  const int n = min(hdr->n_chunks, max_chunks);
  const int lane = threadIdx.x & 31, grp = lane / RL::GS, gl = lane % RL::GS, col = gl * RL::VPL;
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t w = warp; w < n; w += nwarps) {
    const Chunk ch = chunks[w];
    float c[RL::VPL];
    ldg_vec<RL::VPL>(c, C + (int64_t)ch.row * W + col);
    sddmm_range<W>(c, ch.p0, ch.p1, crd, vals, D, Y, grp, col, gl);
  }
}

inline int grid_rows(int64_t nwarps_needed) {
  int64_t ctas = (nwarps_needed + 7) / 8;
  const int64_t cap = (int64_t)device_sm_count() * 32;
  if (ctas > cap) ctas = cap;
  return (int)(ctas < 1 ? 1 : ctas);
}

}  // namespace

cudaError_t launch_sddmm_spmm_rows(const CsrView& B, const float* C, const float* D, int L,
                                   const float* E, int K, float* A, const SplitPlan& plan, cudaStream_t s) {
  if (B.nrows <= 0) return cudaSuccess;
  const int WM = L > K ? L : K;
  // as many CTAs as stay resident; hdr->next_row starts at 0 (header zeroed by the call)
  int64_t ctas = ceil_div(ceil_div(B.nrows, kRowsPerClaim) + plan.max_chunks, 8);
  const int64_t cap = (int64_t)device_sm_count() * SLNR_SDDMM_MIN_CTAS;
  if (ctas > cap) ctas = cap;
  SLNR_WIDTH_SWITCH(WM, W, {
    k_sddmm_spmm_rows<W><<<SLNR_COUNTED((unsigned)ctas), 256, 0, s>>>(plan.hdr, B.nrows, B.pos, B.crd, B.vals, C, D, L, E, K, A,
                                                         plan.chunks, plan.max_chunks, plan.partial);
  });
  return cudaGetLastError();
}

cudaError_t launch_sddmm_spmm_chunks(const CsrView& B, const float* C, const float* D, int L,
                                     const float* E, int K, const SplitPlan& plan, cudaStream_t s) {
  if (plan.max_chunks <= 0) return cudaSuccess;
  const int WM = L > K ? L : K;
  SLNR_WIDTH_SWITCH(WM, W, {
    k_sddmm_spmm_chunks<W><<<SLNR_COUNTED(grid_rows(plan.max_chunks)), 256, 0, s>>>(plan.hdr, plan.chunks, plan.max_chunks,
                                                                      B.crd, B.vals, C, D, L, E, K,
                                                                      plan.partial);
  });
  return cudaGetLastError();
}

cudaError_t launch_sddmm_spmm_gemm_tiles(const CsrView& B, const float* C, const float* D, int K,
                                         const float* F, int L, const float* W, int M, float* A, cudaStream_t s) {
  if (B.nrows <= 0) return cudaSuccess;
  const int64_t grid = ceil_div(B.nrows, kTileRows);
  const size_t smem = tile_smem_bytes(L, M);
  const int WM = K > L ? K : L;
  SLNR_WIDTH_SWITCH(WM, WMC, {
    SLNR_WIDTH_SWITCH(L, LC, {
      if (LC <= WMC) {
        cudaError_t e = set_smem(k_sddmm_spmm_gemm_tiles<WMC, LC <= WMC ? LC : WMC>, smem);
        if (e != cudaSuccess) return e;
        k_sddmm_spmm_gemm_tiles<WMC, LC <= WMC ? LC : WMC><<<SLNR_COUNTED((unsigned)grid), 256, smem, s>>>(
            B.nrows, B.pos, B.crd, B.vals, C, D, K, F, W, M, A);
      }
    });
  });
  return cudaGetLastError();
}

cudaError_t launch_sddmm_rows(const CsrView& B, const float* C, const float* D, int L, float* Y,
                              cudaStream_t s) {
  if (B.nrows <= 0) return cudaSuccess;
  SLNR_WIDTH_SWITCH(L, W, {
    k_sddmm_rows<W><<<SLNR_COUNTED(grid_rows(B.nrows)), 256, 0, s>>>(B.nrows, B.pos, B.crd, B.vals, C, D, Y);
  });
  return cudaGetLastError();
}

cudaError_t launch_sddmm_chunks(const CsrView& B, const float* C, const float* D, int L, float* Y,
                                const SplitPlan& plan, cudaStream_t s) {
  if (plan.max_chunks <= 0) return cudaSuccess;
  SLNR_WIDTH_SWITCH(L, W, {
    k_sddmm_chunks<W><<<SLNR_COUNTED(grid_rows(plan.max_chunks)), 256, 0, s>>>(plan.hdr, plan.chunks, plan.max_chunks,
                                                                 B.crd, B.vals, C, D, Y);
  });
  return cudaGetLastError();
}

}  // namespace slnr
