// Sparse-times-dense producer stages and the heavy-row combine.
//
//   out[r,:] = sum_{p in row r} vals[p] * X[crd[p], :]        (width W)
//
// This is the SpMM of Fig. 2b and the producer of <SpMM,GEMM> (T = B.C),
// of <SpTTM,SpTTM> (T = B x_3 C per fiber) and of MTTKRP's unfused variant.
// A group of lanes owns one row (common.cuh, RowLanes), so light rows need no
// cross-lane reduction; heavy rows go through chunks and k_combine.  With H
// the gathered row is X[k,:] .* X2[k,:] (the producer of <SpMMH,GEMM>).
#include "launch.h"

namespace slnr {
namespace {

template <int W, bool H>
__global__ void __launch_bounds__(256) k_spmm_rows(int nrows, const int32_t* __restrict__ pos,
                                                   const int32_t* __restrict__ crd,
                                                   const float* __restrict__ vals,
                                                   const float* __restrict__ X, const float* __restrict__ X2,
                                                   float* __restrict__ out) {
  using RL = RowLanes<W>;
  const int lane = threadIdx.x & 31, grp = lane / RL::GS, col = (lane % RL::GS) * RL::VPL;
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t r = warp * RL::GPW + grp; r < nrows; r += nwarps * RL::GPW) {
    const int p0 = pos[r], p1 = pos[r + 1];
    if (p1 - p0 > kLightMax) continue;  // written by the heavy-row path
    float acc[RL::VPL];
    zero_vec(acc);
    gather_acc<RL::VPL, H ? 2 : 4, H>(acc, crd, vals, p0, p1, X, W, col, X2);
    st_vec(out + r * W + col, acc);
  }
}

template <int W, bool H>
__global__ void __launch_bounds__(256) k_spmm_chunks(const WsHeader* __restrict__ hdr,
                                                     const Chunk* __restrict__ chunks, int max_chunks,
                                                     const int32_t* __restrict__ crd,
                                                     const float* __restrict__ vals,
                                                     const float* __restrict__ X, const float* __restrict__ X2,
                                                     float* __restrict__ partial) {
  using RL = RowLanes<W>;
  const int n = min(hdr->n_chunks, max_chunks);
  const int lane = threadIdx.x & 31, grp = lane / RL::GS, col = (lane % RL::GS) * RL::VPL;
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t c = warp * RL::GPW + grp; c < n; c += nwarps * RL::GPW) {
    const Chunk ch = chunks[c];
    float acc[RL::VPL];
    zero_vec(acc);
    gather_acc<RL::VPL, H ? 2 : 4, H>(acc, crd, vals, ch.p0, ch.p1, X, W, col, X2);
    st_vec(partial + (int64_t)ch.slot * W + col, acc);
  }
}

// Heavy rows with at most this many partials are summed by one warp when no D
// follows, longer ones by a CTA, both in one launch (k_combine_rows); with D
// every row by a CTA (k_combine).
constexpr int kWarpCombine = 16;

// One CTA per heavy row: the row's partials (width W) are summed by
// kRowLanes lanes each taking every kRowLanes-th partial, then by a fixed
// pairwise tree, so the result does not depend on scheduling and long rows
// keep a short rounding chain.  With D, the sum t (length W = K) is then
// multiplied by D (K x L): out[row, l] = sum_k t[k] D[k, l].  Without D, rows
// of at most kWarpCombine partials are left to the warps of k_combine_rows.
// The CTA's share: heavy rows first, first + stride, ... (block-uniform).
template <int W>
__device__ __forceinline__ void combine_cta(const WsHeader* __restrict__ hdr, const HeavyRow* __restrict__ heavy,
                                            int max_heavy, const float* __restrict__ partial,
                                            const float* __restrict__ D, int L, float* __restrict__ out, int first,
                                            int stride) {
  constexpr int NC = W / 4;                 // float4 columns
  constexpr int NR = 256 / NC;              // lanes along the partials
  __shared__ float4 red[256];
  __shared__ float t[W];
  const int n = min(hdr->n_heavy, max_heavy);
  const int c4 = threadIdx.x % NC, rl = threadIdx.x / NC;
  for (int h = first; h < n; h += stride) {
    const HeavyRow hr = heavy[h];
    if (D == nullptr && hr.count <= kWarpCombine) continue;  // k_combine_rows writes it (block-uniform)
    float4 s = make_float4(0.f, 0.f, 0.f, 0.f);
    if (rl < NR) {
      for (int c = rl; c < hr.count; c += NR) {
        const float4 v = __ldg(reinterpret_cast<const float4*>(partial + (int64_t)(hr.base + c) * W) + c4);
        s.x += v.x; s.y += v.y; s.z += v.z; s.w += v.w;
      }
    }
    red[threadIdx.x] = s;
    __syncthreads();
    for (int half = NR / 2; half > 0; half >>= 1) {
      if (rl < half) {
        const float4 o = red[(rl + half) * NC + c4];
        float4 m = red[rl * NC + c4];
        m.x += o.x; m.y += o.y; m.z += o.z; m.w += o.w;
        red[rl * NC + c4] = m;
      }
      __syncthreads();
    }
    if (D == nullptr) {
      if (rl == 0) reinterpret_cast<float4*>(out + (int64_t)hr.row * W)[c4] = red[c4];
    } else {
      if (rl == 0) {
        const float4 v = red[c4];
        t[4 * c4 + 0] = v.x; t[4 * c4 + 1] = v.y; t[4 * c4 + 2] = v.z; t[4 * c4 + 3] = v.w;
      }
      __syncthreads();
      for (int l = threadIdx.x; l < L; l += blockDim.x) {
        float acc = 0.f;
#pragma unroll 8
        for (int k = 0; k < W; ++k) acc = fmaf(t[k], __ldg(D + (int64_t)k * L + l), acc);
        out[(int64_t)hr.row * L + l] = acc;
      }
    }
    __syncthreads();
  }
}

template <int W>
__global__ void __launch_bounds__(256) k_combine(const WsHeader* __restrict__ hdr,
                                                 const HeavyRow* __restrict__ heavy, int max_heavy,
                                                 const float* __restrict__ partial,
                                                 const float* __restrict__ D, int L,
                                                 float* __restrict__ out) {
  combine_cta<W>(hdr, heavy, max_heavy, partial, D, L, out, blockIdx.x, gridDim.x);
}

// Without D, rows of at most kWarpCombine partials: a warp per heavy row
// (grid-stride), lane l holding the columns [VPL l, VPL l + VPL); the row's
// partials are added in their order (four loads in flight) and the sum
// written.  Deterministic: the order is fixed.  Rows with more partials go to
// the CTAs of combine_cta, whose lanes split them.
template <int W>
__device__ __forceinline__ void combine_warps(const WsHeader* __restrict__ hdr, const HeavyRow* __restrict__ heavy,
                                              int max_heavy, const float* __restrict__ partial,
                                              float* __restrict__ out, int64_t warp, int64_t nwarps) {
  using RL = RowLanes<W>;
  const int n = min(hdr->n_heavy, max_heavy);
  const int lane = threadIdx.x & 31, grp = lane / RL::GS, col = (lane % RL::GS) * RL::VPL;
  for (int64_t h = warp * RL::GPW + grp; h < n; h += nwarps * RL::GPW) {
    const HeavyRow hr = heavy[h];
    if (hr.count > kWarpCombine) continue;
    float acc[RL::VPL];
    zero_vec(acc);
    int c = 0;
    for (; c + 4 <= hr.count; c += 4) {
      float x[4][RL::VPL];
#pragma unroll
      for (int u = 0; u < 4; ++u) ldg_vec<RL::VPL>(x[u], partial + (int64_t)(hr.base + c + u) * W + col);
#pragma unroll
      for (int u = 0; u < 4; ++u)
#pragma unroll
        for (int e = 0; e < RL::VPL; ++e) acc[e] += x[u][e];
    }
    for (; c < hr.count; ++c) {
      float x[RL::VPL];
      ldg_vec<RL::VPL>(x, partial + (int64_t)(hr.base + c) * W + col);
#pragma unroll
      for (int e = 0; e < RL::VPL; ++e) acc[e] += x[e];
    }
    st_vec(out + (int64_t)hr.row * W + col, acc);
  }
}

// Without D, both kinds of heavy row in one launch: the first `nbig` CTAs
// take the rows of more than kWarpCombine partials (a CTA each, as
// k_combine), the other CTAs' warps the rest (a warp each, in order).
template <int W>
__global__ void __launch_bounds__(256) k_combine_rows(const WsHeader* __restrict__ hdr,
                                                      const HeavyRow* __restrict__ heavy, int max_heavy,
                                                      const float* __restrict__ partial, float* __restrict__ out,
                                                      int nbig) {
  if ((int)blockIdx.x < nbig) {
    combine_cta<W>(hdr, heavy, max_heavy, partial, nullptr, 0, out, blockIdx.x, nbig);
    return;
  }
  const int64_t warp = ((int64_t)(blockIdx.x - nbig) * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)(gridDim.x - nbig) * blockDim.x) >> 5;
  combine_warps<W>(hdr, heavy, max_heavy, partial, out, warp, nwarps);
}

inline int grid_warps(int64_t items_per_warp_round, int64_t n) {
  // enough CTAs of 8 warps to cover n items (items_per_warp_round per warp),
  // capped at 32 CTAs per SM; grid-stride loops cover the rest
  int64_t warps = (n + items_per_warp_round - 1) / items_per_warp_round;
  int64_t ctas = (warps + 7) / 8;
  const int64_t cap = (int64_t)device_sm_count() * 32;
  if (ctas > cap) ctas = cap;
  return (int)(ctas < 1 ? 1 : ctas);
}

}  // namespace

cudaError_t launch_spmm_rows(int W, const CsrView& B, const float* X, float* out, cudaStream_t s,
                             const float* X2) {
  if (B.nrows <= 0) return cudaSuccess;
  SLNR_WIDTH_SWITCH(W, WC, {
    const int grid = grid_warps(RowLanes<WC>::GPW, B.nrows);
    if (X2 == nullptr)
      k_spmm_rows<WC, false><<<SLNR_COUNTED(grid), 256, 0, s>>>(B.nrows, B.pos, B.crd, B.vals, X, nullptr, out);
    else
      k_spmm_rows<WC, true><<<SLNR_COUNTED(grid), 256, 0, s>>>(B.nrows, B.pos, B.crd, B.vals, X, X2, out);
  });
  return cudaGetLastError();
}

cudaError_t launch_spmm_chunks(int W, const CsrView& B, const float* X, const SplitPlan& plan,
                               cudaStream_t s, const float* X2) {
  if (plan.max_chunks <= 0) return cudaSuccess;
  SLNR_WIDTH_SWITCH(W, WC, {
    const int grid = grid_warps(RowLanes<WC>::GPW, plan.max_chunks);
    if (X2 == nullptr)
      k_spmm_chunks<WC, false><<<SLNR_COUNTED(grid), 256, 0, s>>>(plan.hdr, plan.chunks, plan.max_chunks, B.crd, B.vals, X,
                                                     nullptr, plan.partial);
    else
      k_spmm_chunks<WC, true><<<SLNR_COUNTED(grid), 256, 0, s>>>(plan.hdr, plan.chunks, plan.max_chunks, B.crd, B.vals, X, X2,
                                                    plan.partial);
  });
  return cudaGetLastError();
}

cudaError_t launch_combine(int W, const SplitPlan& plan, const float* D, int L, float* out,
                           cudaStream_t s) {
  if (plan.max_heavy <= 0) return cudaSuccess;
  int grid = plan.max_heavy;
  const int cap = device_sm_count() * 8;
  if (grid > cap) grid = cap;
  if (D == nullptr) {  // rows with many partials a CTA each, the others a warp each, in one launch
    const int nbig = device_sm_count() * 2 < grid ? device_sm_count() * 2 : grid;
    SLNR_WIDTH_SWITCH(W, WC, {
      k_combine_rows<WC><<<SLNR_COUNTED(nbig + grid_warps(RowLanes<WC>::GPW, plan.max_heavy)), 256, 0, s>>>(
          plan.hdr, plan.heavy, plan.max_heavy, plan.partial, out, nbig);
    });
    return cudaGetLastError();
  }
  SLNR_WIDTH_SWITCH(W, WC, {
    k_combine<WC><<<SLNR_COUNTED(grid), 256, 0, s>>>(plan.hdr, plan.heavy, plan.max_heavy, plan.partial, D, L, out);
  });
  return cudaGetLastError();
}

}  // namespace slnr
