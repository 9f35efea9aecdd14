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
#define SLNR_MTTKRP_MIN_CTAS 5  // resident 256-thread CTAs per SM the unit kernel is compiled for (48 registers)
#endif
#ifndef SLNR_MTTKRP_U
#define SLNR_MTTKRP_U 4  // nonzeros of a fiber in flight per lane group
#endif

namespace slnr {
namespace {

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
  using RL = RowLanes<L>;
  const int n = min(hdr->n_units, max_units);
  const int lane = threadIdx.x & 31, grp = lane / RL::GS, col = (lane % RL::GS) * RL::VPL;
  // warps take units one at a time from the header's counter (units of hub
  // slices hold far more work than those of small slices)
  for (;;) {
    int w = 0;
    if (lane == 0) w = atomicAdd(&hdr->next_unit, 1);
    w = __shfl_sync(0xffffffffu, w, 0);
    if (w >= n) break;
    const Unit un = units[w];
    const int flo = un.flo, fhi = un.fhi;  // fibers starting in the unit's window (inspector)
    float acc[RL::VPL];
    zero_vec(acc);
    // The group's fibers f = flo + grp + n GPW, software-pipelined in three
    // stages so that one round trip serves three fibers: with fiber f's rows
    // in flight, the first nonzero (k, value) of fiber f + GPW and the record
    // (pos3 range, j) of fiber f + 2 GPW are loaded.  Most fibers have one
    // nonzero, whose D row then needs no further dependent load.
    constexpr int GPW = RL::GPW;
    auto load_rec = [&](int f, int& p0, int& p1, int& j) {
      if (f < fhi) { p0 = __ldg(pos3 + f); p1 = __ldg(pos3 + f + 1); j = __ldg(crd2 + f); }
      else { p0 = 0; p1 = 0; j = 0; }
    };
    auto load_first = [&](int p0, int p1, int& k, float& v) {
      if (p0 < p1) { k = __ldg(crd3 + p0); v = __ldg(vals + p0); }
      else { k = -1; v = 0.f; }
    };
    int f = flo + grp;
    int p0a, p1a, ja, p0b, p1b, jb, ka;
    float va;
    load_rec(f, p0a, p1a, ja);
    load_rec(f + GPW, p0b, p1b, jb);
    load_first(p0a, p1a, ka, va);
    for (; f < fhi; f += GPW) {
      int kb, p0c, p1c, jc;
      float vb;
      load_first(p0b, p1b, kb, vb);
      load_rec(f + 2 * GPW, p0c, p1c, jc);
      float c[RL::VPL];
      ldg_vec<RL::VPL>(c, C + (int64_t)ja * L + col);
      // producer: T(l) = sum_k B(i,j,k) D(k,l), in registers, in nonzero order
      float t[RL::VPL];
      zero_vec(t);
      if (ka >= 0) {
        float x[RL::VPL];
        ldg_vec<RL::VPL>(x, D + (int64_t)ka * L + col);
#pragma unroll
        for (int e = 0; e < RL::VPL; ++e) t[e] = fmaf(va, x[e], t[e]);
        gather_acc<RL::VPL, SLNR_MTTKRP_U>(t, crd3, vals, p0a + 1, p1a, D, L, col);
      }
      // consumer: A(i,l) += T(l) C(j,l)
#pragma unroll
      for (int x = 0; x < RL::VPL; ++x) acc[x] = fmaf(t[x], c[x], acc[x]);
      p0a = p0b; p1a = p1b; ja = jb; ka = kb; va = vb;
      p0b = p0c; p1b = p1c; jb = jc;
    }
    cross_group_sum<RL::GS>(acc);
    if (grp == 0) st_vec(partial + w * L + col, acc);
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
    k_mttkrp_units<W><<<ctas, 256, 0, s>>>(plan.hdr, plan.units, plan.slice_units,
                                                                 plan.max_units, B.pos2, B.crd2, B.pos3,
                                                                 B.crd3, B.vals, C, D, plan.partial);
  });
  return cudaGetLastError();
}

cudaError_t launch_mttkrp_stage2_units(int L, const slnr_csf3& B, const float* T, const float* C,
                                       const UnitPlan& plan, cudaStream_t s) {
  if (plan.max_units <= 0 || B.nslices <= 0) return cudaSuccess;
  SLNR_WIDTH_SWITCH(L, W, {
    k_mttkrp_stage2_units<W><<<grid_units(plan.max_units), 256, 0, s>>>(
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
    k_mttkrp_parts<W><<<(unsigned)pgrid, 256, 0, s>>>(plan.hdr, plan.units, plan.slice_units, plan.max_units,
                                                      plan.partial, plan.part_sums);
    k_mttkrp_combine<W><<<(unsigned)grid, 256, 0, s>>>(B.nslices, B.crd1, plan.slice_units, plan.partial,
                                                       plan.part_sums, E, M, A);
  });
  return cudaGetLastError();
}

}  // namespace slnr
