// MTTKRP:  A(i,l) = sum_{j,k} B(i,j,k) * C(j,l) * D(k,l),  B in CSF (i -> j -> k)
// and <MTTKRP,GEMM>: the same followed by A(i,:).E.
//
// Fused schedule (Sec. 4.2, Algorithm 1 removing C): the shared loops are the
// slice i and the fiber j; the producer builds T(l) = sum_k B(i,j,k) D(k,l)
// for one fiber and the consumer adds T .* C(j,:) to A(i,:) at once.  Zipf
// slice sizes put a fifth of all nonzeros in one slice, so each slice is cut
// into units (fibers starting in one window of kUnitNnz nonzeros); a warp
// owns a unit, its lane groups own fibers, and each unit leaves one partial
// A row.  k_mttkrp_combine sums a row's partials in a fixed pairwise order
// and writes every row of A (zero for rows without a slice).
//
// Unfused schedule: T(f,:) for every fiber f is first written to memory
// (spmm.cu over the fiber level), then k_mttkrp_stage2_units reads it.
#include "launch.h"

#ifndef SLNR_MTTKRP_MIN_CTAS
#define SLNR_MTTKRP_MIN_CTAS 4  // resident 256-thread CTAs per SM the unit kernel is compiled for (64 registers)
#endif
#ifndef SLNR_MTTKRP_U
#define SLNR_MTTKRP_U 4  // nonzeros a lane group gathers at once (each a D row and, at a fiber's end, a C row)
#endif

namespace slnr {
namespace {

// Lane layout of the fused unit kernel: a gathered row of L values is read by
// a group of GS lanes (VPL columns each), a warp holds G groups.
template <int L>
struct FlatLanes {
  static constexpr int VPL = L >= 256 ? 8 : 4;
  static constexpr int GS = L / VPL;
  static constexpr int G = 32 / GS;
  static constexpr int B = 32 / G;                       // nonzeros per group per warp step
  static constexpr int UB0 = VPL == 8 ? SLNR_MTTKRP_U / 2 : SLNR_MTTKRP_U;  // same registers for wide rows
  static constexpr int UB = B < UB0 ? B : UB0;           // of those, gathered at once
  static_assert(GS >= 1 && GS <= 32 && B % UB == 0, "lane layout");
};

// Fused MTTKRP over units (windows of at most kUnitNnz consecutive nonzeros
// of one slice), nonzero-parallel: a warp takes a unit and walks its
// nonzeros in steps of 32, lane l holding nonzero q + l (coordinate and
// value loaded coalesced).  The fibers those nonzeros belong to come from a
// coalesced window of the next 32 fiber starts: each lane counts the starts
// at or before its nonzero (a binary search over the window by shuffles), so
// no load waits for another load of the same step.  Lane group g then
// gathers the D rows of nonzeros g B .. g B + B - 1, sums each fiber's run in
// nonzero order (the producer, T(l) = sum_k B(i,j,k) D(k,l)) and, where the
// run ends, multiplies it by C(j,:) and adds it to the unit's partial row
// (the consumer).  A fiber that spans groups or steps contributes one run
// per piece, which by linearity adds up to its T times C(j,:).  The order is
// fixed by the data, so results are the same on every run.
template <int L>
__global__ void __launch_bounds__(256, SLNR_MTTKRP_MIN_CTAS) k_mttkrp_units(WsHeader* __restrict__ hdr,
                                                      const Unit* __restrict__ units,
                                                      const SliceUnits* __restrict__ sus, int max_units,
                                                      const int32_t* __restrict__ pos2,
                                                      const int32_t* __restrict__ crd2,
                                                      const int32_t* __restrict__ pos3,
                                                      const int32_t* __restrict__ crd3,
                                                      const float* __restrict__ vals,
                                                      const float* __restrict__ C,
                                                      const float* __restrict__ D,
                                                      float* __restrict__ partial) {
  using FL = FlatLanes<L>;
  constexpr int VPL = FL::VPL, GS = FL::GS, B = FL::B, UB = FL::UB;
  constexpr unsigned FULL = 0xffffffffu;
  const int n = min(hdr->n_units, max_units);
  const int lane = threadIdx.x & 31, g = lane / GS, col = (lane % GS) * VPL;
  for (;;) {
    int w = 0;
    if (lane == 0) w = atomicAdd(&hdr->next_unit, 1);
    w = __shfl_sync(FULL, w, 0);
    if (w >= n) break;
    const Unit un = units[w];
    const int hi = un.p1, f1 = __ldg(pos2 + un.slice + 1);
    int q = un.p0, fcur = un.ffirst;  // pos3[fcur] <= q
    float acc[VPL];
    zero_vec(acc);
    while (q < hi) {  // warp-uniform
      // the window: starts of fibers fcur + 1 .. fcur + 32 (past the slice: never)
      const int fm = fcur + 1 + lane;
      const int s = fm < f1 ? __ldg(pos3 + fm) : INT_MAX;
      const int jn = fm < f1 ? __ldg(crd2 + fm) : 0;
      const int j0 = __ldg(crd2 + fcur);
      const int qe = min(min(q + 32, hi), __shfl_sync(FULL, s, 31));  // labels stay inside the window
      const int p = q + lane;
      const bool live = p < qe;
      const int kk = live ? __ldg(crd3 + p) : 0;
      const float vv = live ? __ldg(vals + p) : 0.f;
      // cnt = starts at or before p (s is sorted): p is in fiber fcur + cnt
      int cnt = 0;
#pragma unroll
      for (int step = 16; step > 0; step >>= 1)
        if (__shfl_sync(FULL, s, cnt + step - 1) <= p) cnt += step;
      const int jx = __shfl_sync(FULL, jn, cnt > 0 ? cnt - 1 : 0);
      const int jj = cnt > 0 ? jx : j0;
      const int cprev = __shfl_up_sync(FULL, cnt, 1), cnext = __shfl_down_sync(FULL, cnt, 1);
      const bool start = lane % B == 0 || cprev != cnt;
      const bool end = live && (lane % B == B - 1 || p + 1 >= qe || cnext != cnt);
      const int flags = (start ? 1 : 0) | (end ? 2 : 0) | (live ? 4 : 0);
      // group g: its B nonzeros in order, UB at a time
      float t[VPL];
      zero_vec(t);
#pragma unroll
      for (int u0 = 0; u0 < B; u0 += UB) {
        float x[UB][VPL], cr[UB][VPL], v[UB];
        int fl[UB];
#pragma unroll
        for (int k = 0; k < UB; ++k) {
          const int l = g * B + u0 + k;
          const int ck = __shfl_sync(FULL, kk, l), jk = __shfl_sync(FULL, jj, l);
          v[k] = __shfl_sync(FULL, vv, l);
          fl[k] = __shfl_sync(FULL, flags, l);
          if (fl[k] & 4) ldg_vec<VPL>(x[k], D + (int64_t)ck * L + col); else zero_vec(x[k]);
          if (fl[k] & 2) ldg_vec<VPL>(cr[k], C + (int64_t)jk * L + col); else zero_vec(cr[k]);
        }
#pragma unroll
        for (int k = 0; k < UB; ++k) {
#pragma unroll
          for (int e = 0; e < VPL; ++e) t[e] = fmaf(v[k], x[k][e], (fl[k] & 1) ? 0.f : t[e]);
          if (fl[k] & 2)
#pragma unroll
            for (int e = 0; e < VPL; ++e) acc[e] = fmaf(t[e], cr[k][e], acc[e]);
        }
      }
      // the next step starts in the fiber holding qe
      fcur += __popc(__ballot_sync(FULL, s <= qe));
      q = qe;
    }
    cross_group_sum<GS>(acc);
    if (g == 0) st_vec(partial + (int64_t)w * L + col, acc);
  }
}

template <int L>
__global__ void __launch_bounds__(256) k_mttkrp_stage2_units(const WsHeader* __restrict__ hdr,
                                                             const Unit* __restrict__ units,
                                                             const SliceUnits* __restrict__ sus, int max_units,
                                                             const int32_t* __restrict__ pos2,
                                                             const int32_t* __restrict__ crd2,
                                                             const int32_t* __restrict__ pos3,
                                                             const float* __restrict__ T,
                                                             const float* __restrict__ C,
                                                             float* __restrict__ partial) {
  using RL = RowLanes<L>;
  const int n = min(hdr->n_units, max_units);
  const int lane = threadIdx.x & 31, grp = lane / RL::GS, col = (lane % RL::GS) * RL::VPL;
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t w = warp; w < n; w += nwarps) {
    const Unit un = units[w];
    const int flo = un.flo, fhi = un.fhi;  // fibers starting in the unit's window (inspector)
    float acc[RL::VPL];
    zero_vec(acc);
    for (int f = flo + grp; f < fhi; f += RL::GPW) {
      const int j = __ldg(crd2 + f);
      float c[RL::VPL], t[RL::VPL];
      ldg_vec<RL::VPL>(c, C + (int64_t)j * L + col);
      ldg_vec<RL::VPL>(t, T + (int64_t)f * L + col);
#pragma unroll
      for (int x = 0; x < RL::VPL; ++x) acc[x] = fmaf(t[x], c[x], acc[x]);
    }
    cross_group_sum<RL::GS>(acc);
    if (grp == 0) st_vec(partial + w * L + col, acc);
  }
}

// k_mttkrp_combine writes A from the unit partials: slices of more than
// kWarpSlice units are combined by a whole CTA each, the others by one warp
// each, in the same launch (the CTAs holding a hub slice do it first, while
// the rest of the grid takes the small slices).
constexpr int kWarpSlice = 16;

// Warp phase: a warp per slice q (grid-stride) of at most kWarpSlice units: lane row rw
// sums the partials rw, rw + NRW, ... in order, a fixed xor-shuffle tree adds
// the NRW row sums (every lane ends with the same total), and A(crd1[q], :)
// is written; with E (L x M) A(crd1[q], :) = u . E instead, lane m taking
// outputs m, m + 32, ... with u(l) broadcast from the lane holding it.
template <int L>
__device__ __forceinline__ void combine_small_slices(int nslices, const int32_t* __restrict__ crd1,
                                                     const SliceUnits* __restrict__ sus,
                                                     const float* __restrict__ partial,
                                                     const float* __restrict__ E, int M, float* __restrict__ A) {
  constexpr int NC = L / 4;                  // float4 columns of a row
  constexpr int CPL = NC > 32 ? NC / 32 : 1;  // float4 columns per lane
  constexpr int LPR = NC / CPL;               // lanes per row
  constexpr int NRW = 32 / LPR;               // partial rows summed at once
  const int lane = threadIdx.x & 31, c4 = lane % LPR, rw = lane / LPR;
  const int64_t gwarp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t q = gwarp; q < nslices; q += nwarps) {
    const SliceUnits su = sus[q];
    if (su.count > kWarpSlice) continue;  // warp-uniform: k_mttkrp_combine writes it
    const int i = __ldg(crd1 + q);
    float4 s[CPL];
#pragma unroll
    for (int h = 0; h < CPL; ++h) s[h] = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int u = rw; u < su.count; u += NRW) {
      const float4* row = reinterpret_cast<const float4*>(partial + (int64_t)(su.base + u) * L);
#pragma unroll
      for (int h = 0; h < CPL; ++h) {
        const float4 v = __ldg(row + c4 + h * LPR);
        s[h].x += v.x; s[h].y += v.y; s[h].z += v.z; s[h].w += v.w;
      }
    }
#pragma unroll
    for (int off = LPR; off < 32; off <<= 1)
#pragma unroll
      for (int h = 0; h < CPL; ++h) {
        s[h].x += __shfl_xor_sync(0xffffffffu, s[h].x, off);
        s[h].y += __shfl_xor_sync(0xffffffffu, s[h].y, off);
        s[h].z += __shfl_xor_sync(0xffffffffu, s[h].z, off);
        s[h].w += __shfl_xor_sync(0xffffffffu, s[h].w, off);
      }
    if (E == nullptr) {
      if (rw == 0) {
        float4* dst = reinterpret_cast<float4*>(A + (int64_t)i * L);
#pragma unroll
        for (int h = 0; h < CPL; ++h) dst[c4 + h * LPR] = s[h];
      }
    } else {
      for (int m0 = 0; m0 < M; m0 += 32) {  // warp-uniform
        const int m = m0 + lane;
        float acc = 0.f;
#pragma unroll
        for (int l = 0; l < L; ++l) {
          const int f4 = l / 4, h = f4 / LPR;
          const float4 v = s[h];
          const float mine = (l % 4 == 0) ? v.x : (l % 4 == 1) ? v.y : (l % 4 == 2) ? v.z : v.w;
          const float ul = __shfl_sync(0xffffffffu, mine, f4 % LPR);
          if (m < M) acc = fmaf(ul, __ldg(E + (int64_t)l * M + m), acc);
        }
        if (m < M) A[(int64_t)i * M + m] = acc;
      }
    }
  }
}

// A slice of more than kWarpSlice units is summed in two levels: runs of
// kPartUnits consecutive unit partials first (k_mttkrp_parts, a warp per run,
// so a hub slice of thousands of units spreads over the GPU), then its part
// sums by one CTA (k_mttkrp_combine).  Both levels add in a fixed order.
constexpr int kPartUnits = 64;

// A warp per run: each lane checks one unit, the run leaders (unit u of a
// large slice with u a multiple of kPartUnits) are taken in turn by the whole
// warp.  Lane row rw adds the run's partials rw, rw + NRW, ... in order, a
// fixed xor-shuffle tree adds the row sums, and the sum is written to
// part_sums row base + u / kPartUnits (inside the slice's own unit range).
template <int L>
__global__ void __launch_bounds__(256) k_mttkrp_parts(const WsHeader* __restrict__ hdr,
                                                      const Unit* __restrict__ units,
                                                      const SliceUnits* __restrict__ sus, int max_units,
                                                      const float* __restrict__ partial,
                                                      float* __restrict__ part_sums) {
  constexpr int NC = L / 4;
  constexpr int CPL = NC > 32 ? NC / 32 : 1;
  constexpr int LPR = NC / CPL;
  constexpr int NRW = 32 / LPR;
  const int n = min(hdr->n_units, max_units);
  const int lane = threadIdx.x & 31, c4 = lane % LPR, rw = lane / LPR;
  const int64_t gwarp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t w0 = gwarp * 32; w0 < n; w0 += nwarps * 32) {
    bool lead = false;
    if (w0 + lane < n) {
      const Unit un = units[w0 + lane];
      lead = un.u % kPartUnits == 0 && sus[un.slice].count > kWarpSlice;
    }
    unsigned m = __ballot_sync(0xffffffffu, lead);
    while (m != 0) {  // warp-uniform
      const int b = __ffs(m) - 1;
      m &= m - 1;
      const Unit un = units[w0 + b];
      const SliceUnits su = sus[un.slice];
      const int u1 = min(un.u + kPartUnits, su.count);
      float4 s[CPL];
#pragma unroll
      for (int h = 0; h < CPL; ++h) s[h] = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 4
      for (int u = un.u + rw; u < u1; u += NRW) {
        const float4* row = reinterpret_cast<const float4*>(partial + (int64_t)(su.base + u) * L);
#pragma unroll
        for (int h = 0; h < CPL; ++h) {
          const float4 v = __ldg(row + c4 + h * LPR);
          s[h].x += v.x; s[h].y += v.y; s[h].z += v.z; s[h].w += v.w;
        }
      }
#pragma unroll
      for (int off = LPR; off < 32; off <<= 1)
#pragma unroll
        for (int h = 0; h < CPL; ++h) {
          s[h].x += __shfl_xor_sync(0xffffffffu, s[h].x, off);
          s[h].y += __shfl_xor_sync(0xffffffffu, s[h].y, off);
          s[h].z += __shfl_xor_sync(0xffffffffu, s[h].z, off);
          s[h].w += __shfl_xor_sync(0xffffffffu, s[h].w, off);
        }
      if (rw == 0) {
        float4* dst = reinterpret_cast<float4*>(part_sums + (int64_t)(su.base + un.u / kPartUnits) * L);
#pragma unroll
        for (int h = 0; h < CPL; ++h) dst[c4 + h * LPR] = s[h];
      }
    }
  }
}

// CTA phase, then the warp phase.  CTA phase: one CTA per slice q of more
// than kWarpSlice units (grid-stride over chunks of the slices; a chunk's
// large slices are listed first, one load per thread): sums the slice's part
// sums (strided lanes, each adding in order, then a fixed pairwise tree) and
// writes A(crd1[q], :).
// Rows of A without a slice were zero-filled before the launch.  With E
// (L x M, <MTTKRP,GEMM>) the row u(i,:) stays in shared memory and
// A(i,:) = u(i,:).E is written instead (width M): the MTTKRP result is never
// stored.
template <int L>
__global__ void __launch_bounds__(256) k_mttkrp_combine(int nslices, const int32_t* __restrict__ crd1,
                                                        const SliceUnits* __restrict__ sus,
                                                        const float* __restrict__ partial,
                                                        const float* __restrict__ part_sums,
                                                        const float* __restrict__ E, int M,
                                                        float* __restrict__ A) {
  constexpr int NC = L / 4;
  constexpr int NR = 256 / NC;
  __shared__ float4 red[256];
  __shared__ int big[256];
  __shared__ int nbig;
  const int c4 = threadIdx.x % NC, rl = threadIdx.x / NC;
  for (int64_t base = blockIdx.x; base < nslices; base += (int64_t)gridDim.x * 256) {
    if (threadIdx.x == 0) nbig = 0;
    __syncthreads();
    const int64_t qt = base + (int64_t)threadIdx.x * gridDim.x;
    if (qt < nslices && sus[qt].count > kWarpSlice) big[atomicAdd(&nbig, 1)] = (int)qt;
    __syncthreads();
    const int nb = nbig;
    for (int b = 0; b < nb; ++b) {
      const int q = big[b];
      const int i = __ldg(crd1 + q);
      const SliceUnits su = sus[q];
      const int np = (su.count + kPartUnits - 1) / kPartUnits;  // its part sums (k_mttkrp_parts)
      float4 s = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 4
      for (int u = rl; u < np; u += NR) {
        const float4 v = __ldg(reinterpret_cast<const float4*>(part_sums + (int64_t)(su.base + u) * L) + c4);
        s.x += v.x; s.y += v.y; s.z += v.z; s.w += v.w;
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
      if (E == nullptr) {
        if (rl == 0) reinterpret_cast<float4*>(A + (int64_t)i * L)[c4] = red[c4];
      } else {
        const float* uu = reinterpret_cast<const float*>(red);  // u(i,0..L)
        for (int m = threadIdx.x; m < M; m += blockDim.x) {
          float acc = 0.f;
#pragma unroll 8
          for (int l = 0; l < L; ++l) acc = fmaf(uu[l], __ldg(E + (int64_t)l * M + m), acc);
          A[(int64_t)i * M + m] = acc;
        }
      }
      __syncthreads();
    }
    __syncthreads();  // every thread has read nbig before the next chunk resets it
  }
  combine_small_slices<L>(nslices, crd1, sus, partial, E, M, A);
}

inline int grid_units(int64_t max_units) {
  int64_t ctas = (max_units + 7) / 8;
  const int64_t cap = (int64_t)device_sm_count() * 32;
  if (ctas > cap) ctas = cap;
  return (int)(ctas < 1 ? 1 : ctas);
}

}  // namespace

cudaError_t launch_mttkrp_units(int L, const slnr_csf3& B, const float* C, const float* D,
                                const UnitPlan& plan, cudaStream_t s) {
  if (plan.max_units <= 0 || B.nslices <= 0) return cudaSuccess;
  SLNR_WIDTH_SWITCH(L, W, {
    int ctas = grid_units(plan.max_units);  // as many as stay resident: warps take units dynamically
    if (ctas > device_sm_count() * SLNR_MTTKRP_MIN_CTAS) ctas = device_sm_count() * SLNR_MTTKRP_MIN_CTAS;
    k_mttkrp_units<W><<<SLNR_COUNTED(ctas), 256, 0, s>>>(plan.hdr, plan.units, plan.slice_units,
                                                                 plan.max_units, B.pos2, B.crd2, B.pos3,
                                                                 B.crd3, B.vals, C, D, plan.partial);
  });
  return cudaGetLastError();
}

cudaError_t launch_mttkrp_stage2_units(int L, const slnr_csf3& B, const float* T, const float* C,
                                       const UnitPlan& plan, cudaStream_t s) {
  if (plan.max_units <= 0 || B.nslices <= 0) return cudaSuccess;
  SLNR_WIDTH_SWITCH(L, W, {
    k_mttkrp_stage2_units<W><<<SLNR_COUNTED(grid_units(plan.max_units)), 256, 0, s>>>(
        plan.hdr, plan.units, plan.slice_units, plan.max_units, B.pos2, B.crd2, B.pos3, T, C, plan.partial);
  });
  return cudaGetLastError();
}

cudaError_t launch_mttkrp_combine(int L, const slnr_csf3& B, const UnitPlan& plan, const float* E, int M,
                                  float* A, cudaStream_t s) {
  if (B.dim[0] <= 0) return cudaSuccess;
  // rows of A without a slice are zero; the kernel writes the others
  cudaError_t e = cudaMemsetAsync(A, 0, sizeof(float) * (size_t)B.dim[0] * (size_t)(E != nullptr ? M : L), s);
  if (e != cudaSuccess || B.nslices <= 0) return e;
  // a warp per slice in the warp phase (8 per CTA); grid-stride beyond
  int64_t grid = ceil_div(B.nslices, 8);
  if (grid > (int64_t)device_sm_count() * 32) grid = (int64_t)device_sm_count() * 32;
  SLNR_WIDTH_SWITCH(L, W, {
    int64_t pgrid = ceil_div(plan.max_units, 32 * 8);  // a warp per 32 units
    if (pgrid > (int64_t)device_sm_count() * 32) pgrid = (int64_t)device_sm_count() * 32;
    k_mttkrp_parts<W><<<SLNR_COUNTED((unsigned)pgrid), 256, 0, s>>>(plan.hdr, plan.units, plan.slice_units, plan.max_units,
                                                      plan.partial, plan.part_sums);
    k_mttkrp_combine<W><<<SLNR_COUNTED((unsigned)grid), 256, 0, s>>>(B.nslices, B.crd1, plan.slice_units, plan.partial,
                                                       plan.part_sums, E, M, A);
  });
  return cudaGetLastError();
}

}  // namespace slnr
