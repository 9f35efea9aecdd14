// Kernels for inner dimensions outside the specialised ones: any multiple of
// 4 up to kWideMax (1024).  The specialised kernels take powers of two in
// [4, 256] with lane layouts fixed at compile time; these take the width at
// run time.
//
// Lane layout: a warp owns a row; lane l holds the float4 columns
// l, l + 32, ..., l + 32 (NCH - 1) of it (NCH = ceil(W / 128), a template
// parameter in {1, 2, 4, 8}), columns past W masked off.  The schedules are
// the same as the specialised kernels': fused variants keep the temporary
// (T row, or scalar per stored (i,j)) on chip, heavy rows are cut into chunks
// whose partial rows are summed in a fixed order, and every sum runs in a
// fixed order (results are the same on every run).
#include "launch.h"

namespace slnr {
namespace {

constexpr int kWTileRows = 32;  // rows of a CTA's T tile (fused tile kernels, dense GEMM)
constexpr int kWKChunk = 32;    // rows of the consumer matrix staged per step
constexpr int kWThreads = 256;

template <int NCH>
__device__ __forceinline__ void wzero(float4 (&a)[NCH]) {
#pragma unroll
  for (int i = 0; i < NCH; ++i) a[i] = make_float4(0.f, 0.f, 0.f, 0.f);
}

// a = row[lane's columns] (0 past W)
template <int NCH>
__device__ __forceinline__ void wload(float4 (&a)[NCH], const float* __restrict__ row, int W, int lane) {
#pragma unroll
  for (int i = 0; i < NCH; ++i) {
    const int c4 = lane + 32 * i;
    a[i] = 4 * c4 < W ? __ldg(reinterpret_cast<const float4*>(row) + c4) : make_float4(0.f, 0.f, 0.f, 0.f);
  }
}

template <int NCH>
__device__ __forceinline__ void wstore(float* row, const float4 (&a)[NCH], int W, int lane) {
#pragma unroll
  for (int i = 0; i < NCH; ++i) {
    const int c4 = lane + 32 * i;
    if (4 * c4 < W) reinterpret_cast<float4*>(row)[c4] = a[i];
  }
}

__device__ __forceinline__ void fma4(float4& a, float s, const float4& x) {
  a.x = fmaf(s, x.x, a.x);
  a.y = fmaf(s, x.y, a.y);
  a.z = fmaf(s, x.z, a.z);
  a.w = fmaf(s, x.w, a.w);
}

__device__ __forceinline__ float4 mul4(const float4& a, const float4& b) {
  return make_float4(a.x * b.x, a.y * b.y, a.z * b.z, a.w * b.w);
}

// acc = sum_{p in [p0,p1)} vals[p] R(crd[p]), in p order, two rows in flight;
// R(k) = X[k,:] (width W), or X[k,:] .* X2[k,:] with H.
template <int NCH, bool H>
__device__ __forceinline__ void wgather(float4 (&acc)[NCH], const int32_t* __restrict__ crd,
                                        const float* __restrict__ vals, int p0, int p1, const float* __restrict__ X,
                                        const float* __restrict__ X2, int W, int lane) {
  wzero(acc);
  int p = p0;
  for (; p + 2 <= p1; p += 2) {
    const int c0 = __ldg(crd + p), c1 = __ldg(crd + p + 1);
    const float v0 = __ldg(vals + p), v1 = __ldg(vals + p + 1);
    float4 x0[NCH], x1[NCH];
    wload(x0, X + (int64_t)c0 * W, W, lane);
    wload(x1, X + (int64_t)c1 * W, W, lane);
    if constexpr (H) {
      float4 y0[NCH], y1[NCH];
      wload(y0, X2 + (int64_t)c0 * W, W, lane);
      wload(y1, X2 + (int64_t)c1 * W, W, lane);
#pragma unroll
      for (int i = 0; i < NCH; ++i) {
        x0[i] = mul4(x0[i], y0[i]);
        x1[i] = mul4(x1[i], y1[i]);
      }
    }
#pragma unroll
    for (int i = 0; i < NCH; ++i) fma4(acc[i], v0, x0[i]);
#pragma unroll
    for (int i = 0; i < NCH; ++i) fma4(acc[i], v1, x1[i]);
  }
  if (p < p1) {
    const int c0 = __ldg(crd + p);
    const float v0 = __ldg(vals + p);
    float4 x0[NCH];
    wload(x0, X + (int64_t)c0 * W, W, lane);
    if constexpr (H) {
      float4 y0[NCH];
      wload(y0, X2 + (int64_t)c0 * W, W, lane);
#pragma unroll
      for (int i = 0; i < NCH; ++i) x0[i] = mul4(x0[i], y0[i]);
    }
#pragma unroll
    for (int i = 0; i < NCH; ++i) fma4(acc[i], v0, x0[i]);
  }
}

// out[r,:] = sum_p vals[p] R(crd[p]) for every light row r, and the partial
// rows of heavy-row chunks: a warp per item, the chunks first (grid-stride
// over n_chunks + nrows items; with out NULL, the chunks only).  Producer of the unfused <SpMM,GEMM>,
// <SpTTM,SpTTM>, <SpMMH,GEMM> and MTTKRP, and of the second step of the
// unfused <SDDMM,SpMM> (vals = the sampled products).
template <int NCH, bool H>
__global__ void __launch_bounds__(kWThreads) k_w_spmm(const WsHeader* __restrict__ hdr, int nrows,
                                                      const int32_t* __restrict__ pos,
                                                      const int32_t* __restrict__ crd,
                                                      const float* __restrict__ vals, const float* __restrict__ X,
                                                      const float* __restrict__ X2, int W, float* __restrict__ out,
                                                      const Chunk* __restrict__ chunks, int max_chunks,
                                                      float* __restrict__ partial) {
  const int lane = threadIdx.x & 31;
  const int nch = min(hdr->n_chunks, max_chunks);
  const int64_t nitems = (int64_t)nch + (out != nullptr ? nrows : 0);  // out NULL: the chunks only
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t w = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; w < nitems; w += nwarps) {
    float4 acc[NCH];
    if (w < nch) {
      const Chunk ch = chunks[w];
      wgather<NCH, H>(acc, crd, vals, ch.p0, ch.p1, X, X2, W, lane);
      wstore(partial + (int64_t)ch.slot * W, acc, W, lane);
    } else {
      const int64_t r = w - nch;
      const int p0 = pos[r], p1 = pos[r + 1];
      if (p1 - p0 > kLightMax) continue;  // its chunks above
      wgather<NCH, H>(acc, crd, vals, p0, p1, X, X2, W, lane);
      wstore(out + r * W, acc, W, lane);
    }
  }
}

// Heavy rows: a warp per row sums the row's partials (width W) in chunk order;
// without D the sum is the row of out (width W); with D (W x L) the sum is
// staged in shared memory and out's row (width L) is sum . D.
template <int NCH>
__global__ void __launch_bounds__(kWThreads) k_w_combine(const WsHeader* __restrict__ hdr,
                                                         const HeavyRow* __restrict__ heavy, int max_heavy,
                                                         const float* __restrict__ partial, int W,
                                                         const float* __restrict__ D, int L, float* __restrict__ out) {
  extern __shared__ float4 wsm4[];
  const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
  float* t = reinterpret_cast<float*>(wsm4) + (size_t)wib * W;  // this warp's row (with D)
  const int n = min(hdr->n_heavy, max_heavy);
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t h = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; h < n; h += nwarps) {
    const HeavyRow hr = heavy[h];
    float4 s[NCH];
    wzero(s);
    for (int c = 0; c < hr.count; ++c) {
      float4 x[NCH];
      wload(x, partial + (int64_t)(hr.base + c) * W, W, lane);
#pragma unroll
      for (int i = 0; i < NCH; ++i) {
        s[i].x += x[i].x;
        s[i].y += x[i].y;
        s[i].z += x[i].z;
        s[i].w += x[i].w;
      }
    }
    if (D == nullptr) {
      wstore(out + (int64_t)hr.row * W, s, W, lane);
      continue;
    }
    __syncwarp();
#pragma unroll
    for (int i = 0; i < NCH; ++i)
      if (4 * (lane + 32 * i) < W) reinterpret_cast<float4*>(t)[lane + 32 * i] = s[i];
    __syncwarp();
    for (int l4 = lane; 4 * l4 < L; l4 += 32) {  // out(row, 4 l4 .. 4 l4 + 3) = t . D, k in order
      float4 a = make_float4(0.f, 0.f, 0.f, 0.f);
      for (int k = 0; k < W; ++k) fma4(a, t[k], __ldg(reinterpret_cast<const float4*>(D + (int64_t)k * L) + l4));
      reinterpret_cast<float4*>(out + (int64_t)hr.row * L)[l4] = a;
    }
  }
}

// Shared memory of the tile kernels: the T tile (kWTileRows x W), the staged
// consumer rows (kWKChunk x 128) and the keep flags.
inline size_t wtile_smem(int W) {
  return sizeof(float) * ((size_t)kWTileRows * W + (size_t)kWKChunk * 128);
}

// The consumer of a T tile in shared memory (kWTileRows rows, width W):
// A(r0 + r, :) = T(r, :) . D for the tile's rows r < nrows - r0 with keep[r]
// (D is W x L).  Warp w computes rows 4w .. 4w + 3, lane l the float4
// column l of each 128-column block; D is staged kWKChunk rows at a time and
// every output is a k-ordered fp32 FMA chain.
__device__ __forceinline__ void wtile_times_d(const float* T, int W, const float* __restrict__ D, int L,
                                              float* Ds, float* __restrict__ A, int64_t r0, int64_t nrows,
                                              const int* keep) {
  const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
  for (int cb = 0; cb < L; cb += 128) {
    float4 acc[4];
#pragma unroll
    for (int r = 0; r < 4; ++r) acc[r] = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int k0 = 0; k0 < W; k0 += kWKChunk) {
      __syncthreads();
      for (int i = threadIdx.x; i < kWKChunk * 32; i += blockDim.x) {
        const int kk = i / 32, c4 = i % 32, k = k0 + kk, c = cb + 4 * c4;
        reinterpret_cast<float4*>(Ds)[i] = (k < W && c < L)
                                               ? __ldg(reinterpret_cast<const float4*>(D + (int64_t)k * L + c))
                                               : make_float4(0.f, 0.f, 0.f, 0.f);
      }
      __syncthreads();
      const int kn = min(kWKChunk, W - k0);
      for (int kk = 0; kk < kn; ++kk) {
        const float4 d = reinterpret_cast<const float4*>(Ds)[kk * 32 + lane];
#pragma unroll
        for (int r = 0; r < 4; ++r) fma4(acc[r], T[(4 * wib + r) * W + k0 + kk], d);
      }
    }
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      const int rr = 4 * wib + r;
      const int64_t row = r0 + rr;
      if (row < nrows && (keep == nullptr || keep[rr]) && cb + 4 * lane < L)
        reinterpret_cast<float4*>(A + row * L + cb)[lane] = acc[r];
    }
  }
}

// Fused <SpMM,GEMM> (and <SpTTM,SpTTM> over fibers, <SpMMH,GEMM> with H) for
// light rows: a CTA owns kWTileRows consecutive rows; warp w builds the T rows
// 4w .. 4w + 3 (T(i,:) = sum_j B(i,j) C(j,:), width K) into the shared tile,
// never to global memory, then the tile is multiplied by D and A's rows are
// written once.  Heavy rows are left to the chunks and the combine (times D).
template <int NCH, bool H>
__global__ void __launch_bounds__(kWThreads) k_w_spmm_gemm_tiles(int nrows, const int32_t* __restrict__ pos,
                                                                 const int32_t* __restrict__ crd,
                                                                 const float* __restrict__ vals,
                                                                 const float* __restrict__ C,
                                                                 const float* __restrict__ C2, int K,
                                                                 const float* __restrict__ D, int L,
                                                                 float* __restrict__ A) {
  extern __shared__ float4 wsm4[];
  float* T = reinterpret_cast<float*>(wsm4);
  float* Ds = T + (size_t)kWTileRows * K;
  __shared__ int keep[kWTileRows];
  const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
  const int64_t r0 = (int64_t)blockIdx.x * kWTileRows;
#pragma unroll 1
  for (int r = 0; r < 4; ++r) {
    const int rr = 4 * wib + r;
    const int64_t row = r0 + rr;
    float4 acc[NCH];
    wzero(acc);
    int ok = 0;
    if (row < nrows) {
      const int p0 = pos[row], p1 = pos[row + 1];
      if (p1 - p0 <= kLightMax) {  // warp-uniform
        wgather<NCH, H>(acc, crd, vals, p0, p1, C, C2, K, lane);
        ok = 1;
      }
    }
#pragma unroll
    for (int i = 0; i < NCH; ++i)
      if (4 * (lane + 32 * i) < K) reinterpret_cast<float4*>(T + (size_t)rr * K)[lane + 32 * i] = acc[i];
    if (lane == 0) keep[rr] = ok;
  }
  wtile_times_d(T, K, D, L, Ds, A, r0, nrows, keep);
}

// Dense A = T . D (M x K times K x L) for the unfused variants: a CTA loads a
// tile of kWTileRows rows of T into shared memory, then the tile consumer.
__global__ void __launch_bounds__(kWThreads) k_w_dense_gemm(int64_t M, const float* __restrict__ Tg, int K,
                                                            const float* __restrict__ D, int L,
                                                            float* __restrict__ A) {
  extern __shared__ float4 wsm4[];
  float* T = reinterpret_cast<float*>(wsm4);
  float* Ds = T + (size_t)kWTileRows * K;
  const int64_t r0 = (int64_t)blockIdx.x * kWTileRows;
  for (int i = threadIdx.x; i < kWTileRows * (K / 4); i += blockDim.x) {
    const int rr = i / (K / 4), c4 = i % (K / 4);
    reinterpret_cast<float4*>(T)[i] = r0 + rr < M ? __ldg(reinterpret_cast<const float4*>(Tg + (r0 + rr) * K) + c4)
                                                  : make_float4(0.f, 0.f, 0.f, 0.f);
  }
  wtile_times_d(T, K, D, L, Ds, A, r0, M, nullptr);
}

// <SDDMM,SpMM> row work: for each nonzero p in [p0, p1) in order,
//   y = vals[p] <c, D(crd[p], :)>   (width Kd; c = C(i,:) staged in shared memory)
//   acc += y E(crd[p], :)           (width Ko)
// two nonzeros in flight; the dot products are warp reductions in a fixed
// xor order.  With Y not NULL the scalars are written to Y[p] instead and acc
// is left alone (the unfused first step).
template <int NCH>
__device__ __forceinline__ void w_sddmm_row(float4 (&acc)[NCH], const float* cs, int p0, int p1,
                                            const int32_t* __restrict__ crd, const float* __restrict__ vals,
                                            const float* __restrict__ D, int Kd, const float* __restrict__ E,
                                            int Ko, float* __restrict__ Y, int lane) {
  float4 c[NCH];
#pragma unroll
  for (int i = 0; i < NCH; ++i)
    c[i] = 4 * (lane + 32 * i) < Kd ? reinterpret_cast<const float4*>(cs)[lane + 32 * i]
                                     : make_float4(0.f, 0.f, 0.f, 0.f);
  for (int p = p0; p < p1; p += 2) {
    const bool two = p + 1 < p1;
    const int j0 = __ldg(crd + p), j1 = two ? __ldg(crd + p + 1) : j0;
    float4 d0[NCH], d1[NCH];
    wload(d0, D + (int64_t)j0 * Kd, Kd, lane);
    wload(d1, D + (int64_t)j1 * Kd, Kd, lane);
    float s0 = 0.f, s1 = 0.f;
#pragma unroll
    for (int i = 0; i < NCH; ++i) {
      s0 = fmaf(c[i].x, d0[i].x, s0); s0 = fmaf(c[i].y, d0[i].y, s0);
      s0 = fmaf(c[i].z, d0[i].z, s0); s0 = fmaf(c[i].w, d0[i].w, s0);
      s1 = fmaf(c[i].x, d1[i].x, s1); s1 = fmaf(c[i].y, d1[i].y, s1);
      s1 = fmaf(c[i].z, d1[i].z, s1); s1 = fmaf(c[i].w, d1[i].w, s1);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      s0 += __shfl_xor_sync(0xffffffffu, s0, o);
      s1 += __shfl_xor_sync(0xffffffffu, s1, o);
    }
    const float y0 = __ldg(vals + p) * s0, y1 = two ? __ldg(vals + p + 1) * s1 : 0.f;
    if (Y != nullptr) {
      if (lane == 0) {
        Y[p] = y0;
        if (two) Y[p + 1] = y1;
      }
      continue;
    }
    float4 e0[NCH], e1[NCH];
    wload(e0, E + (int64_t)j0 * Ko, Ko, lane);
    if (two) wload(e1, E + (int64_t)j1 * Ko, Ko, lane); else wzero(e1);
#pragma unroll
    for (int i = 0; i < NCH; ++i) fma4(acc[i], y0, e0[i]);
    if (two)
#pragma unroll
      for (int i = 0; i < NCH; ++i) fma4(acc[i], y1, e1[i]);
  }
}

// Stages C(row, :) (width Kd) in this warp's shared row cs.
__device__ __forceinline__ void w_stage_row(float* cs, const float* __restrict__ C, int64_t row, int Kd, int lane) {
  __syncwarp();
  for (int c4 = lane; 4 * c4 < Kd; c4 += 32)
    reinterpret_cast<float4*>(cs)[c4] = __ldg(reinterpret_cast<const float4*>(C + row * Kd) + c4);
  __syncwarp();
}

// Fused <SDDMM,SpMM> (A(i,:) = sum_j B(i,j) <C(i,:), D(j,:)> E(j,:)): a warp
// per item, heavy-row chunks first (partial rows of width Ko), then light
// rows (A rows written once; with A NULL, the chunks only).  With Y not NULL:
// the unfused first step, the sampled products Y[p] for every nonzero.
template <int NCH>
__global__ void __launch_bounds__(kWThreads) k_w_sddmm_spmm(const WsHeader* __restrict__ hdr, int nrows,
                                                            const int32_t* __restrict__ pos,
                                                            const int32_t* __restrict__ crd,
                                                            const float* __restrict__ vals,
                                                            const float* __restrict__ C, const float* __restrict__ D,
                                                            int Kd, const float* __restrict__ E, int Ko,
                                                            float* __restrict__ A, const Chunk* __restrict__ chunks,
                                                            int max_chunks, float* __restrict__ partial,
                                                            float* __restrict__ Y) {
  extern __shared__ float4 wsm4[];
  const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
  float* cs = reinterpret_cast<float*>(wsm4) + (size_t)wib * Kd;
  const int nch = min(hdr->n_chunks, max_chunks);
  const int64_t nitems = (int64_t)nch + (A != nullptr || Y != nullptr ? nrows : 0);  // A, Y NULL: the chunks only
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t w = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; w < nitems; w += nwarps) {
    float4 acc[NCH];
    wzero(acc);
    if (w < nch) {
      const Chunk ch = chunks[w];
      w_stage_row(cs, C, ch.row, Kd, lane);
      w_sddmm_row<NCH>(acc, cs, ch.p0, ch.p1, crd, vals, D, Kd, E, Ko, Y, lane);
      if (Y == nullptr) wstore(partial + (int64_t)ch.slot * Ko, acc, Ko, lane);
    } else {
      const int64_t r = w - nch;
      const int p0 = pos[r], p1 = pos[r + 1];
      if (p1 - p0 > kLightMax) continue;  // its chunks above
      w_stage_row(cs, C, r, Kd, lane);
      w_sddmm_row<NCH>(acc, cs, p0, p1, crd, vals, D, Kd, E, Ko, Y, lane);
      if (Y == nullptr) wstore(A + r * Ko, acc, Ko, lane);
    }
  }
}

// Fused <SDDMM,SpMM,GEMM> over light rows (Algorithm 1 applied twice): a CTA
// owns kWTileRows rows; warp w builds the vector temporaries
// T(i,:) = sum_j B(i,j) <C(i,:), D(j,:)> F(j,:) (width L) of rows 4w .. 4w + 3
// into the shared tile, then the tile is multiplied by W (L x M).  Heavy rows
// go through k_w_sddmm_spmm's chunks and the combine (times W).
template <int NCH>
__global__ void __launch_bounds__(kWThreads) k_w_sddmm_spmm_gemm_tiles(int nrows, const int32_t* __restrict__ pos,
                                                                       const int32_t* __restrict__ crd,
                                                                       const float* __restrict__ vals,
                                                                       const float* __restrict__ C,
                                                                       const float* __restrict__ D, int K,
                                                                       const float* __restrict__ F, int L,
                                                                       const float* __restrict__ Wm, int M,
                                                                       float* __restrict__ A) {
  extern __shared__ float4 wsm4[];
  float* T = reinterpret_cast<float*>(wsm4);
  float* Ds = T + (size_t)kWTileRows * L;
  float* cs = Ds + (size_t)kWKChunk * 128 + (size_t)(threadIdx.x >> 5) * K;
  __shared__ int keep[kWTileRows];
  const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
  const int64_t r0 = (int64_t)blockIdx.x * kWTileRows;
#pragma unroll 1
  for (int r = 0; r < 4; ++r) {
    const int rr = 4 * wib + r;
    const int64_t row = r0 + rr;
    float4 acc[NCH];
    wzero(acc);
    int ok = 0;
    if (row < nrows) {
      const int p0 = pos[row], p1 = pos[row + 1];
      if (p1 - p0 <= kLightMax) {  // warp-uniform
        w_stage_row(cs, C, row, K, lane);
        w_sddmm_row<NCH>(acc, cs, p0, p1, crd, vals, D, K, F, L, nullptr, lane);
        ok = 1;
      }
    }
#pragma unroll
    for (int i = 0; i < NCH; ++i)
      if (4 * (lane + 32 * i) < L) reinterpret_cast<float4*>(T + (size_t)rr * L)[lane + 32 * i] = acc[i];
    if (lane == 0) keep[rr] = ok;
  }
  wtile_times_d(T, L, Wm, M, Ds, A, r0, nrows, keep);
}

// MTTKRP over units (the fibers of a slice that start in one window of
// kUnitNnz nonzeros): a warp per unit, its fibers in order; per fiber the
// producer T(l) = sum_k B(i,j,k) D(k,l) (or, unfused, T's row read from
// memory) and the consumer acc += T .* C(j,:); one partial row per unit.
template <int NCH, bool TG>
__global__ void __launch_bounds__(kWThreads) k_w_mttkrp_units(const WsHeader* __restrict__ hdr,
                                                              const Unit* __restrict__ units, int max_units,
                                                              const int32_t* __restrict__ crd2,
                                                              const int32_t* __restrict__ pos3,
                                                              const int32_t* __restrict__ crd3,
                                                              const float* __restrict__ vals,
                                                              const float* __restrict__ C,
                                                              const float* __restrict__ D,
                                                              const float* __restrict__ Tg, int L,
                                                              float* __restrict__ partial) {
  const int lane = threadIdx.x & 31;
  const int n = min(hdr->n_units, max_units);
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t w = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; w < n; w += nwarps) {
    const Unit un = units[w];
    float4 acc[NCH];
    wzero(acc);
    for (int f = un.flo; f < un.fhi; ++f) {
      const int j = __ldg(crd2 + f);
      float4 t[NCH], c[NCH];
      if constexpr (TG)
        wload(t, Tg + (int64_t)f * L, L, lane);
      else
        wgather<NCH, false>(t, crd3, vals, __ldg(pos3 + f), __ldg(pos3 + f + 1), D, nullptr, L, lane);
      wload(c, C + (int64_t)j * L, L, lane);
#pragma unroll
      for (int i = 0; i < NCH; ++i) {
        acc[i].x = fmaf(t[i].x, c[i].x, acc[i].x);
        acc[i].y = fmaf(t[i].y, c[i].y, acc[i].y);
        acc[i].z = fmaf(t[i].z, c[i].z, acc[i].z);
        acc[i].w = fmaf(t[i].w, c[i].w, acc[i].w);
      }
    }
    wstore(partial + w * L, acc, L, lane);
  }
}

// A(i,:) = the sum of slice i's unit partials (width L), a warp per slice,
// units in order; with E (L x M) the sum is staged in shared memory and
// A(i,:) = sum . E (width M).  Rows of A without a slice are zeroed before.
template <int NCH>
__global__ void __launch_bounds__(kWThreads) k_w_mttkrp_combine(int nslices, const int32_t* __restrict__ crd1,
                                                                const SliceUnits* __restrict__ sus,
                                                                const float* __restrict__ partial, int L,
                                                                const float* __restrict__ E, int M,
                                                                float* __restrict__ A) {
  extern __shared__ float4 wsm4[];
  const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
  float* u = reinterpret_cast<float*>(wsm4) + (size_t)wib * L;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t q = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; q < nslices; q += nwarps) {
    const SliceUnits su = sus[q];
    const int i = __ldg(crd1 + q);
    float4 s[NCH];
    wzero(s);
    for (int k = 0; k < su.count; ++k) {
      float4 x[NCH];
      wload(x, partial + (int64_t)(su.base + k) * L, L, lane);
#pragma unroll
      for (int h = 0; h < NCH; ++h) {
        s[h].x += x[h].x;
        s[h].y += x[h].y;
        s[h].z += x[h].z;
        s[h].w += x[h].w;
      }
    }
    if (E == nullptr) {
      wstore(A + (int64_t)i * L, s, L, lane);
      continue;
    }
    __syncwarp();
#pragma unroll
    for (int h = 0; h < NCH; ++h)
      if (4 * (lane + 32 * h) < L) reinterpret_cast<float4*>(u)[lane + 32 * h] = s[h];
    __syncwarp();
    for (int m4 = lane; 4 * m4 < M; m4 += 32) {
      float4 a = make_float4(0.f, 0.f, 0.f, 0.f);
      for (int l = 0; l < L; ++l) fma4(a, u[l], __ldg(reinterpret_cast<const float4*>(E + (int64_t)l * M) + m4));
      reinterpret_cast<float4*>(A + (int64_t)i * M)[m4] = a;
    }
  }
}

// float4 columns per lane for widths up to w: ceil(w / 128) rounded up to 1, 2, 4 or 8
#define SLNR_NCH_SWITCH(w, NC, ...)                                   \
  do {                                                                \
    const int nch_ = ((w) + 127) / 128;                               \
    if (nch_ <= 1) { constexpr int NC = 1; __VA_ARGS__; }             \
    else if (nch_ <= 2) { constexpr int NC = 2; __VA_ARGS__; }        \
    else if (nch_ <= 4) { constexpr int NC = 4; __VA_ARGS__; }        \
    else if (nch_ <= 8) { constexpr int NC = 8; __VA_ARGS__; }        \
    else return cudaErrorInvalidValue;                                \
  } while (0)

inline unsigned w_grid(int64_t items) {  // a warp per item, grid-stride beyond 16 CTAs per SM
  int64_t ctas = (items + 7) / 8;
  const int64_t cap = (int64_t)device_sm_count() * 16;
  if (ctas > cap) ctas = cap;
  return (unsigned)(ctas < 1 ? 1 : ctas);
}

// Opts the kernel in to `bytes` of dynamic shared memory (the default limit
// counts the kernel's static shared memory too, so set it whenever any is asked).
template <typename Kern>
cudaError_t w_smem(Kern k, size_t bytes) {
  if (bytes == 0) return cudaSuccess;
  return cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
}

}  // namespace

bool wide_dim(int d) { return d >= 4 && d <= kWideMax && d % 4 == 0; }

cudaError_t launch_w_spmm(int W, const CsrView& B, const float* X, const float* X2, float* out,
                          const SplitPlan& plan, cudaStream_t s) {
  if (B.nrows <= 0) return cudaSuccess;
  const unsigned grid = w_grid((int64_t)B.nrows + plan.max_chunks);
  SLNR_NCH_SWITCH(W, NC, {
    if (X2 == nullptr)
      k_w_spmm<NC, false><<<SLNR_COUNTED(grid), kWThreads, 0, s>>>(plan.hdr, B.nrows, B.pos, B.crd, B.vals, X, nullptr, W, out,
                                                     plan.chunks, plan.max_chunks, plan.partial);
    else
      k_w_spmm<NC, true><<<SLNR_COUNTED(grid), kWThreads, 0, s>>>(plan.hdr, B.nrows, B.pos, B.crd, B.vals, X, X2, W, out,
                                                    plan.chunks, plan.max_chunks, plan.partial);
  });
  return cudaGetLastError();
}

cudaError_t launch_w_combine(int W, const SplitPlan& plan, const float* D, int L, float* out, cudaStream_t s) {
  if (plan.max_heavy <= 0) return cudaSuccess;
  const size_t smem = D != nullptr ? sizeof(float) * (kWThreads / 32) * (size_t)W : 0;
  SLNR_NCH_SWITCH(W, NC, {
    cudaError_t e = w_smem(k_w_combine<NC>, smem);
    if (e != cudaSuccess) return e;
    k_w_combine<NC><<<SLNR_COUNTED(w_grid(plan.max_heavy)), kWThreads, smem, s>>>(plan.hdr, plan.heavy, plan.max_heavy,
                                                                     plan.partial, W, D, L, out);
  });
  return cudaGetLastError();
}

cudaError_t launch_w_spmm_gemm_tiles(int K, int L, const CsrView& B, const float* C, const float* C2,
                                     const float* D, float* A, cudaStream_t s) {
  if (B.nrows <= 0) return cudaSuccess;
  const int64_t grid = ceil_div(B.nrows, kWTileRows);
  const size_t smem = wtile_smem(K);
  SLNR_NCH_SWITCH(K, NC, {
    if (C2 == nullptr) {
      cudaError_t e = w_smem(k_w_spmm_gemm_tiles<NC, false>, smem);
      if (e != cudaSuccess) return e;
      k_w_spmm_gemm_tiles<NC, false><<<SLNR_COUNTED((unsigned)grid), kWThreads, smem, s>>>(B.nrows, B.pos, B.crd, B.vals, C,
                                                                             nullptr, K, D, L, A);
    } else {
      cudaError_t e = w_smem(k_w_spmm_gemm_tiles<NC, true>, smem);
      if (e != cudaSuccess) return e;
      k_w_spmm_gemm_tiles<NC, true><<<SLNR_COUNTED((unsigned)grid), kWThreads, smem, s>>>(B.nrows, B.pos, B.crd, B.vals, C, C2,
                                                                            K, D, L, A);
    }
  });
  return cudaGetLastError();
}

cudaError_t launch_w_dense_gemm(int64_t M, int K, int L, const float* T, const float* D, float* A, cudaStream_t s) {
  if (M <= 0) return cudaSuccess;
  const size_t smem = wtile_smem(K);
  cudaError_t e = w_smem(k_w_dense_gemm, smem);
  if (e != cudaSuccess) return e;
  k_w_dense_gemm<<<SLNR_COUNTED((unsigned)ceil_div(M, kWTileRows)), kWThreads, smem, s>>>(M, T, K, D, L, A);
  return cudaGetLastError();
}

cudaError_t launch_w_sddmm_spmm(const CsrView& B, const float* C, const float* D, int Kd, const float* E, int Ko,
                                float* A, float* Y, const SplitPlan& plan, cudaStream_t s) {
  if (B.nrows <= 0) return cudaSuccess;
  const size_t smem = sizeof(float) * (kWThreads / 32) * (size_t)Kd;
  const int wmax = Kd > Ko ? Kd : Ko;
  SLNR_NCH_SWITCH(wmax, NC, {
    cudaError_t e = w_smem(k_w_sddmm_spmm<NC>, smem);
    if (e != cudaSuccess) return e;
    k_w_sddmm_spmm<NC><<<SLNR_COUNTED(w_grid((int64_t)B.nrows + plan.max_chunks)), kWThreads, smem, s>>>(
        plan.hdr, B.nrows, B.pos, B.crd, B.vals, C, D, Kd, E, Ko, A, plan.chunks, plan.max_chunks, plan.partial, Y);
  });
  return cudaGetLastError();
}

cudaError_t launch_w_sddmm_spmm_gemm_tiles(const CsrView& B, const float* C, const float* D, int K, const float* F,
                                           int L, const float* W, int M, float* A, cudaStream_t s) {
  if (B.nrows <= 0) return cudaSuccess;
  const size_t smem = wtile_smem(L) + sizeof(float) * (kWThreads / 32) * (size_t)K;
  const int wmax = K > L ? K : L;
  SLNR_NCH_SWITCH(wmax, NC, {
    cudaError_t e = w_smem(k_w_sddmm_spmm_gemm_tiles<NC>, smem);
    if (e != cudaSuccess) return e;
    k_w_sddmm_spmm_gemm_tiles<NC><<<SLNR_COUNTED((unsigned)ceil_div(B.nrows, kWTileRows)), kWThreads, smem, s>>>(
        B.nrows, B.pos, B.crd, B.vals, C, D, K, F, L, W, M, A);
  });
  return cudaGetLastError();
}

cudaError_t launch_w_mttkrp_units(int L, const slnr_csf3& B, const float* C, const float* D, const float* T,
                                  const UnitPlan& plan, cudaStream_t s) {
  if (plan.max_units <= 0 || B.nslices <= 0) return cudaSuccess;
  const unsigned grid = w_grid(plan.max_units);
  SLNR_NCH_SWITCH(L, NC, {
    if (T == nullptr)
      k_w_mttkrp_units<NC, false><<<SLNR_COUNTED(grid), kWThreads, 0, s>>>(plan.hdr, plan.units, plan.max_units, B.crd2, B.pos3,
                                                             B.crd3, B.vals, C, D, nullptr, L, plan.partial);
    else
      k_w_mttkrp_units<NC, true><<<SLNR_COUNTED(grid), kWThreads, 0, s>>>(plan.hdr, plan.units, plan.max_units, B.crd2, B.pos3,
                                                            B.crd3, B.vals, C, D, T, L, plan.partial);
  });
  return cudaGetLastError();
}

cudaError_t launch_w_mttkrp_combine(int L, const slnr_csf3& B, const UnitPlan& plan, const float* E, int M, float* A,
                                    cudaStream_t s) {
  if (B.dim[0] <= 0) return cudaSuccess;
  cudaError_t e = cudaMemsetAsync(A, 0, sizeof(float) * (size_t)B.dim[0] * (size_t)(E != nullptr ? M : L), s);
  if (e != cudaSuccess || B.nslices <= 0) return e;
  const size_t smem = E != nullptr ? sizeof(float) * (kWThreads / 32) * (size_t)L : 0;
  SLNR_NCH_SWITCH(L, NC, {
    e = w_smem(k_w_mttkrp_combine<NC>, smem);
    if (e != cudaSuccess) return e;
    k_w_mttkrp_combine<NC><<<SLNR_COUNTED(w_grid(B.nslices)), kWThreads, smem, s>>>(B.nslices, B.crd1, plan.slice_units,
                                                                        plan.partial, L, E, M, A);
  });
  return cudaGetLastError();
}

}  // namespace slnr
