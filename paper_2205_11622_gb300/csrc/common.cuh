// Shared device-side pieces of libslnr: work-item records written by the
// inspector kernels, lane layouts for gathering dense rows, and the vector
// gather-accumulate loop that every producer stage is built from.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "slnr.h"

namespace slnr {

// ---------------------------------------------------------------------------
// Row splitting ("inspector").  Power-law inputs have rows (or fibers) with
// tens of thousands of nonzeros next to empty ones (load imbalance is the
// second challenge named in Sec. 1).  A row with more than kLightMax nonzeros
// is "heavy": it is cut into chunks of at most kChunk nonzeros, each chunk
// produces a partial row in the workspace, and a combine kernel sums the
// partials of a row in a fixed order (deterministic results).
constexpr int kLightMax = 256;
constexpr int kChunk = 256;
// MTTKRP: a slice is cut into units of fibers that start within one window
// of kUnitNnz nonzeros.
constexpr int kUnitNnz = 512;
// Tensor-core path: rows are cut into segments of at most kSegChunk nonzeros,
// listed by length class (kSegClasses classes: (64,128], (32,64], ..., 2, 1,
// empty); the inspector keeps kSegCounters counters per block of rows (one
// per class, heavy rows, chunks of heavy rows).
constexpr int kSegChunk = 128;
constexpr int kSegClasses = 9;
constexpr int kSegCounters = kSegClasses + 2;

struct WsHeader {        // first 256 bytes of every workspace
  int n_heavy;           // heavy rows found by the inspector
  int n_chunks;          // chunks of heavy rows
  int n_units;           // MTTKRP units
  int error;             // validation / runtime flags (bit set = problem found)
  int n_segs;            // segments of the tensor-core path
  int next_tile;         // tensor-core path: next item tile to hand to a CTA
  int next_row;          // fused <SDDMM,SpMM>: next block of rows to hand to a warp
  int next_unit;         // fused MTTKRP: next unit to hand to a warp
  int pad[56];
};
static_assert(sizeof(WsHeader) == 256, "header is 256 bytes");

struct HeavyRow {        // one heavy row and the slots of its partials
  int row;
  int base;              // first partial slot
  int count;             // number of chunks / partial slots
  int pad;
};

struct Chunk {           // nonzeros [p0, p1) of row `row`, partial goes to `slot`
  int row;
  int p0;
  int p1;
  int slot;
};

struct SliceUnits {      // MTTKRP: units of one slice
  int base;
  int count;
};

struct Unit {            // MTTKRP: window `u` of slice `slice`
  int slice;
  int u;
  int flo;               // fibers starting in the window: [flo, fhi)
  int fhi;
  int p0;                // the window's nonzeros: [p0, p1)
  int p1;
  int ffirst;            // the fiber holding nonzero p0 (the last whose first nonzero is <= p0)
  int pad;
};

// Validation flag bits
enum : int {
  kErrPos = 1,          // position array not monotone / wrong ends
  kErrCrdRange = 2,     // coordinate out of range
  kErrCrdOrder = 4,     // coordinates not strictly increasing in a parent
  kErrOverflow = 8,     // inspector found more work than its bound (malformed positions)
  kErrTimeout = 16,     // a bounded device-side wait gave up
};

// ---------------------------------------------------------------------------
// Lane layout for a dense row of W fp32 values (W a power of two, 4..256):
// a "group" of GS lanes covers one row, each lane VPL consecutive values
// (one or two 16-byte loads), so a group reads the row with fully used
// 32-byte sectors; GPW groups share a warp.
template <int W>
struct RowLanes {
  static_assert(W >= 4 && W <= 256 && (W & (W - 1)) == 0, "W must be a power of two in [4, 256]");
  static constexpr int VPL = (W >= 8) ? 8 : 4;
  static constexpr int GS = W / VPL;
  static constexpr int GPW = 32 / GS;
};

template <int VPL>
__device__ __forceinline__ void ldg_vec(float (&v)[VPL], const float* __restrict__ p) {
  static_assert(VPL % 4 == 0, "whole float4s");
  const float4* q = reinterpret_cast<const float4*>(p);
#pragma unroll
  for (int h = 0; h < VPL / 4; ++h) {
    const float4 a = __ldg(q + h);
    v[4 * h] = a.x; v[4 * h + 1] = a.y; v[4 * h + 2] = a.z; v[4 * h + 3] = a.w;
  }
}

// Loads min(VPL, avail) values (avail is a multiple of 4; the rest are 0).
// Used when one operand of a pair is narrower than the lane layout.
template <int VPL>
__device__ __forceinline__ void ldg_vec_upto(float (&v)[VPL], const float* __restrict__ p, int avail) {
  const float4* q = reinterpret_cast<const float4*>(p);
  float4 a = avail >= 4 ? __ldg(q) : make_float4(0.f, 0.f, 0.f, 0.f);
  v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
  if constexpr (VPL == 8) {
    float4 b = avail >= 8 ? __ldg(q + 1) : make_float4(0.f, 0.f, 0.f, 0.f);
    v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
  }
}

// Stores min(VPL, avail) values (avail a multiple of 4).
template <int VPL>
__device__ __forceinline__ void st_vec_upto(float* p, const float (&v)[VPL], int avail) {
  float4* q = reinterpret_cast<float4*>(p);
  if (avail >= 4) q[0] = make_float4(v[0], v[1], v[2], v[3]);
  if constexpr (VPL == 8)
    if (avail >= 8) q[1] = make_float4(v[4], v[5], v[6], v[7]);
}

template <int VPL>
__device__ __forceinline__ void st_vec(float* p, const float (&v)[VPL]) {
  float4* q = reinterpret_cast<float4*>(p);
  q[0] = make_float4(v[0], v[1], v[2], v[3]);
  if constexpr (VPL == 8) q[1] = make_float4(v[4], v[5], v[6], v[7]);
}

template <int VPL>
__device__ __forceinline__ void zero_vec(float (&v)[VPL]) {
#pragma unroll
  for (int e = 0; e < VPL; ++e) v[e] = 0.f;
}

// acc += sum_{p in [p0,p1)} vals[p] * X[crd[p], col .. col+VPL)
// Sequential in p for every element (fixed order).  U independent row loads
// are in flight per step.  With H (the Hadamard gather of <SpMMH,GEMM>) the
// gathered row is X[crd[p], :] .* X2[crd[p], :], the product formed in fp32
// before the multiply-add.
template <int VPL, int U = 4, bool H = false>
__device__ __forceinline__ void gather_acc(float (&acc)[VPL], const int32_t* __restrict__ crd,
                                           const float* __restrict__ vals, int p0, int p1,
                                           const float* __restrict__ X, int ldx, int col,
                                           const float* __restrict__ X2 = nullptr) {
  int p = p0;
  for (; p + U <= p1; p += U) {
    int c[U];
    float v[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      c[u] = __ldg(crd + p + u);
      v[u] = __ldg(vals + p + u);
    }
    float x[U][VPL];
#pragma unroll
    for (int u = 0; u < U; ++u) ldg_vec<VPL>(x[u], X + (int64_t)c[u] * ldx + col);
    if constexpr (H) {
      float x2[U][VPL];
#pragma unroll
      for (int u = 0; u < U; ++u) ldg_vec<VPL>(x2[u], X2 + (int64_t)c[u] * ldx + col);
#pragma unroll
      for (int u = 0; u < U; ++u)
#pragma unroll
        for (int e = 0; e < VPL; ++e) x[u][e] *= x2[u][e];
    }
#pragma unroll
    for (int u = 0; u < U; ++u)
#pragma unroll
      for (int e = 0; e < VPL; ++e) acc[e] = fmaf(v[u], x[u][e], acc[e]);
  }
  for (; p < p1; ++p) {
    const int c = __ldg(crd + p);
    const float v = __ldg(vals + p);
    float x[VPL];
    ldg_vec<VPL>(x, X + (int64_t)c * ldx + col);
    if constexpr (H) {
      float x2[VPL];
      ldg_vec<VPL>(x2, X2 + (int64_t)c * ldx + col);
#pragma unroll
      for (int e = 0; e < VPL; ++e) x[e] *= x2[e];
    }
#pragma unroll
    for (int e = 0; e < VPL; ++e) acc[e] = fmaf(v, x[e], acc[e]);
  }
}

// Sum of v over the GS lanes of a group (GS a power of two, groups aligned).
template <int GS>
__device__ __forceinline__ float group_sum(float v) {
#pragma unroll
  for (int o = GS / 2; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Elementwise sum of acc across the GPW groups of a warp (result in every group).
template <int GS, int VPL>
__device__ __forceinline__ void cross_group_sum(float (&acc)[VPL]) {
#pragma unroll
  for (int o = GS; o < 32; o <<= 1)
#pragma unroll
    for (int e = 0; e < VPL; ++e) acc[e] += __shfl_xor_sync(0xffffffffu, acc[e], o);
}

__host__ __device__ inline int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }

}  // namespace slnr
