// <SpMM,GEMM> / <SpTTM,SpTTM> with the consumer contraction on tcgen05 TF32
// tensor cores.
//
// Fused schedule (Sec. 4.2, Algorithm 1; the temporary is a vector over k,
// Sec. 6.3): for each row r, T(r,:) = sum_p vals[p] C(crd[p],:) is built on
// chip and A(r,:) = T(r,:) . D follows at once.  Rows are grouped into
// "segments" of at most kSegChunk nonzeros (a row with more nonzeros becomes
// several chunk segments); a persistent CTA takes 128 segments at a time:
//   producer: 16 warps gather C rows into registers and write the 128 x K
//             tile of T, rounded to tf32, into shared memory (128B-swizzled,
//             K-major) -- T never goes to global memory;
//   MMA:      one thread issues K/8 tcgen05.mma (M=128, N=L, K=8) with D^T,
//             staged once per CTA, as the B operand; the fp32 accumulator
//             lives in tensor memory;
//   epilogue: each warp reads its TMEM lane quadrant and writes A rows
//             (whole-row segments) or partial A rows (chunks of heavy rows).
// k_combine (spmm.cu) then sums each heavy row's partial A rows in a fixed
// order: A(r,:) = sum_chunks T_chunk . D, which is exact by linearity.
//
// The same kernel in DENSE mode multiplies a materialised T (unfused
// variant) by D: the producer reads T rows instead of gathering them.
#include "launch.h"
#include "tcgen05.cuh"

namespace slnr {

namespace {

constexpr int kTcThreads = 512;
constexpr int kTcRows = 128;  // MMA M
constexpr int kScanRows = 2048;
constexpr int kScanThreads = 256;
constexpr int kRowsPerThread = kScanRows / kScanThreads;
constexpr long long kWaitCycles = 4000000000LL;  // ~2 s at 2 GHz

__device__ __forceinline__ int segs_of(int n) { return n <= kSegChunk ? 1 : (n + kSegChunk - 1) / kSegChunk; }

// Inclusive block scan of 3 ints (kScanThreads threads); returns block totals in tot.
__device__ __forceinline__ void block_scan3(int (&v)[3], int (&tot)[3]) {
  __shared__ int wsum[kScanThreads / 32][3];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int q = 0; q < 3; ++q)
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, v[q], o);
      if (lane >= o) v[q] += y;
    }
  if (lane == 31)
#pragma unroll
    for (int q = 0; q < 3; ++q) wsum[warp][q] = v[q];
  __syncthreads();
#pragma unroll
  for (int q = 0; q < 3; ++q) {
    int before = 0, all = 0;
    for (int w = 0; w < kScanThreads / 32; ++w) {
      if (w < warp) before += wsum[w][q];
      all += wsum[w][q];
    }
    v[q] += before;
    tot[q] = all;
  }
  __syncthreads();
}

// Pass 1: per block of kScanRows rows, the number of segments, heavy rows and
// heavy-row chunks.
__global__ void __launch_bounds__(kScanThreads) k_seg_count(int nrows, const int32_t* __restrict__ pos,
                                                            int* __restrict__ counts) {
  const int64_t r0 = (int64_t)blockIdx.x * kScanRows + (int64_t)threadIdx.x * kRowsPerThread;
  int v[3] = {0, 0, 0};
  for (int i = 0; i < kRowsPerThread; ++i) {
    const int64_t r = r0 + i;
    if (r < nrows) {
      const int ns = segs_of(pos[r + 1] - pos[r]);
      v[0] += ns;
      if (ns > 1) {
        v[1] += 1;
        v[2] += ns;
      }
    }
  }
  int tot[3];
  block_scan3(v, tot);
  if (threadIdx.x == 0) {
    counts[3 * blockIdx.x + 0] = tot[0];
    counts[3 * blockIdx.x + 1] = tot[1];
    counts[3 * blockIdx.x + 2] = tot[2];
  }
}

// Pass 2: each block adds up the counts of the blocks before it, scans its
// rows and writes their segments (in row order), heavy-row records and chunk
// slots.  The last block publishes the totals in the workspace header.
__global__ void __launch_bounds__(kScanThreads) k_seg_write(int nrows, const int32_t* __restrict__ pos,
                                                            const int* __restrict__ counts, int nblocks,
                                                            WsHeader* hdr, int4* __restrict__ segs,
                                                            HeavyRow* __restrict__ heavy, int max_segs,
                                                            int max_heavy, int max_chunks) {
  __shared__ int base[3];
  if (threadIdx.x < 3) base[threadIdx.x] = 0;
  __syncthreads();
  int pre[3] = {0, 0, 0};
  for (int b = threadIdx.x; b < (int)blockIdx.x; b += blockDim.x) {
    pre[0] += counts[3 * b + 0];
    pre[1] += counts[3 * b + 1];
    pre[2] += counts[3 * b + 2];
  }
#pragma unroll
  for (int q = 0; q < 3; ++q) {
    int x = pre[q];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    if ((threadIdx.x & 31) == 0 && x != 0) atomicAdd(&base[q], x);
  }
  __syncthreads();
  const int64_t r0 = (int64_t)blockIdx.x * kScanRows + (int64_t)threadIdx.x * kRowsPerThread;
  int v[3] = {0, 0, 0};
  for (int i = 0; i < kRowsPerThread; ++i) {
    const int64_t r = r0 + i;
    if (r < nrows) {
      const int ns = segs_of(pos[r + 1] - pos[r]);
      v[0] += ns;
      if (ns > 1) {
        v[1] += 1;
        v[2] += ns;
      }
    }
  }
  const int mine[3] = {v[0], v[1], v[2]};
  int tot[3];
  block_scan3(v, tot);
  int so = base[0] + v[0] - mine[0], ho = base[1] + v[1] - mine[1], co = base[2] + v[2] - mine[2];
  for (int i = 0; i < kRowsPerThread; ++i) {
    const int64_t r = r0 + i;
    if (r >= nrows) break;
    const int p0 = pos[r], p1 = pos[r + 1];
    const int ns = segs_of(p1 - p0);
    if (ns == 1) {
      if (so < max_segs) segs[so] = make_int4((int)r, p0, p1, -1);
      ++so;
    } else {
      if (ho < max_heavy && co + ns <= max_chunks) heavy[ho] = HeavyRow{(int)r, co, ns, 0};
      ++ho;
      for (int c = 0; c < ns; ++c) {
        const int a = p0 + c * kSegChunk;
        if (so < max_segs && co < max_chunks) segs[so] = make_int4((int)r, a, min(p1, a + kSegChunk), co);
        ++so;
        ++co;
      }
    }
  }
  if (blockIdx.x == nblocks - 1 && threadIdx.x == 0) {
    const int ns = base[0] + tot[0], nh = base[1] + tot[1], nc = base[2] + tot[2];
    hdr->n_segs = ns;
    hdr->n_heavy = nh;
    hdr->n_chunks = nc;
    if (ns > max_segs || nh > max_heavy || nc > max_chunks) atomicOr(&hdr->error, kErrOverflow);
  }
}

__device__ __forceinline__ bool mbar_wait_timeout(uint64_t* bar, uint32_t parity) {
  const long long t0 = clock64();
  while (!tc::mbar_try_wait(bar, parity))
    if (clock64() - t0 > kWaitCycles) return false;
  return true;
}

enum TcMode { kSegments = 0, kDense = 1 };

// Shared memory: T tile (kTcRows x K) and D^T (L x K), both tf32 K-major
// 128B-swizzled, plus 1 KB of alignment slack.
__host__ __device__ constexpr size_t tc_smem_bytes(int K, int L) {
  return (size_t)kTcRows * K * 4 + (size_t)L * K * 4 + 1024;
}

template <int K, int L, int MODE>
__global__ void __launch_bounds__(kTcThreads, 1)
    k_tc_gemm(WsHeader* hdr, const int4* __restrict__ segs, int max_segs,
              int64_t dense_rows, const int32_t* __restrict__ crd, const float* __restrict__ vals,
              const float* __restrict__ X, const float* __restrict__ D, float* __restrict__ A,
              float* __restrict__ partial) {
  static_assert(K % 32 == 0 && K >= 32 && K <= 128, "K must be 32, 64 or 128");
  static_assert(L % 32 == 0 && L >= 32 && L <= 256, "L must be a multiple of 32 in [32, 256]");
  constexpr int GS = K / 8;            // lanes per row; each lane: two float4 at k0 and k0 + K/2
  constexpr int GPW = 32 / GS;         // rows per warp pass
  constexpr int NWARPS = kTcThreads / 32;
  constexpr uint32_t IDESC = tc::idesc_tf32(kTcRows, L);
  constexpr uint32_t NCOLS = L;        // TMEM columns of the fp32 accumulator
  extern __shared__ uint8_t smem_raw[];
  __shared__ uint64_t mbar;
  __shared__ uint32_t tmem_base;
  uint8_t* sT = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sD = sT + kTcRows * K * 4;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (warp == 0) {
    tc::tmem_alloc(&tmem_base, NCOLS);
    tc::tmem_relinquish();
  }
  if (tid == 0) {
    tc::mbar_init(&mbar, 1);
    tc::fence_mbar_init();
  }
  // D (K x L, row-major) -> D^T as the B operand (L rows of K), tf32
  for (int i = tid; i < K * (L / 4); i += kTcThreads) {
    const int k = i / (L / 4), n4 = i % (L / 4);
    const float4 d = __ldg(reinterpret_cast<const float4*>(D + (int64_t)k * L) + n4);
    const float dv[4] = {d.x, d.y, d.z, d.w};
#pragma unroll
    for (int e = 0; e < 4; ++e)
      *reinterpret_cast<uint32_t*>(sD + tc::sw128_offset(4 * n4 + e, k, L)) = tc::to_tf32(dv[e]);
  }
  tc::fence_proxy_async_smem();
  tc::tc_fence_before_sync();
  __syncthreads();
  tc::tc_fence_after_sync();
  const uint32_t tmem = tmem_base;
  const uint32_t sT_addr = tc::smem_u32(sT), sD_addr = tc::smem_u32(sD);

  int64_t nitems;
  if (MODE == kSegments) {
    const int n = hdr->n_segs;
    nitems = n < max_segs ? n : max_segs;
  } else {
    nitems = dense_rows;
  }
  const int64_t ntiles = (nitems + kTcRows - 1) / kTcRows;
  const int grp = lane / GS, gl = lane % GS;
  const int k0 = 4 * gl, k1 = 4 * gl + K / 2;
  uint32_t phase = 0;
  bool failed = false;

  for (int64_t t = blockIdx.x; t < ntiles; t += gridDim.x) {
    // ---- producer: T rows of the tile, tf32, swizzled, in shared memory
    for (int s = warp * GPW + grp; s < kTcRows; s += NWARPS * GPW) {
      const int64_t item = t * kTcRows + s;
      float a[4] = {0.f, 0.f, 0.f, 0.f}, b[4] = {0.f, 0.f, 0.f, 0.f};
      if (item < nitems) {
        if (MODE == kSegments) {
          const int4 sg = __ldg(segs + item);
          int p = sg.y;
          const int p1 = sg.z;
          for (; p + 4 <= p1; p += 4) {
            int c[4];
            float v[4];
            float4 x0[4], x1[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
              c[u] = __ldg(crd + p + u);
              v[u] = __ldg(vals + p + u);
            }
#pragma unroll
            for (int u = 0; u < 4; ++u) {
              const float* row = X + (int64_t)c[u] * K;
              x0[u] = __ldg(reinterpret_cast<const float4*>(row + k0));
              x1[u] = __ldg(reinterpret_cast<const float4*>(row + k1));
            }
#pragma unroll
            for (int u = 0; u < 4; ++u) {
              a[0] = fmaf(v[u], x0[u].x, a[0]); a[1] = fmaf(v[u], x0[u].y, a[1]);
              a[2] = fmaf(v[u], x0[u].z, a[2]); a[3] = fmaf(v[u], x0[u].w, a[3]);
              b[0] = fmaf(v[u], x1[u].x, b[0]); b[1] = fmaf(v[u], x1[u].y, b[1]);
              b[2] = fmaf(v[u], x1[u].z, b[2]); b[3] = fmaf(v[u], x1[u].w, b[3]);
            }
          }
          for (; p < p1; ++p) {
            const int c = __ldg(crd + p);
            const float v = __ldg(vals + p);
            const float* row = X + (int64_t)c * K;
            const float4 x0 = __ldg(reinterpret_cast<const float4*>(row + k0));
            const float4 x1 = __ldg(reinterpret_cast<const float4*>(row + k1));
            a[0] = fmaf(v, x0.x, a[0]); a[1] = fmaf(v, x0.y, a[1]); a[2] = fmaf(v, x0.z, a[2]); a[3] = fmaf(v, x0.w, a[3]);
            b[0] = fmaf(v, x1.x, b[0]); b[1] = fmaf(v, x1.y, b[1]); b[2] = fmaf(v, x1.z, b[2]); b[3] = fmaf(v, x1.w, b[3]);
          }
        } else {
          const float* row = X + item * K;
          const float4 x0 = __ldg(reinterpret_cast<const float4*>(row + k0));
          const float4 x1 = __ldg(reinterpret_cast<const float4*>(row + k1));
          a[0] = x0.x; a[1] = x0.y; a[2] = x0.z; a[3] = x0.w;
          b[0] = x1.x; b[1] = x1.y; b[2] = x1.z; b[3] = x1.w;
        }
      }
      *reinterpret_cast<uint4*>(sT + tc::sw128_offset(s, k0, kTcRows)) =
          make_uint4(tc::to_tf32(a[0]), tc::to_tf32(a[1]), tc::to_tf32(a[2]), tc::to_tf32(a[3]));
      *reinterpret_cast<uint4*>(sT + tc::sw128_offset(s, k1, kTcRows)) =
          make_uint4(tc::to_tf32(b[0]), tc::to_tf32(b[1]), tc::to_tf32(b[2]), tc::to_tf32(b[3]));
    }
    tc::fence_proxy_async_smem();
    tc::tc_fence_before_sync();
    __syncthreads();
    // ---- MMA: one thread issues the tile's K/8 steps, then commits to mbar
    if (tid == 0) {
      tc::tc_fence_after_sync();
#pragma unroll
      for (int kb = 0; kb < K / 32; ++kb)
#pragma unroll
        for (int ks = 0; ks < 4; ++ks) {
          const uint64_t ad = tc::desc_k_sw128(sT_addr + kb * kTcRows * 128 + ks * 32);
          const uint64_t bd = tc::desc_k_sw128(sD_addr + kb * L * 128 + ks * 32);
          tc::mma_tf32(tmem, ad, bd, IDESC, (kb | ks) != 0);
        }
      tc::mma_commit(&mbar);
    }
    const bool ok = mbar_wait_timeout(&mbar, phase);
    phase ^= 1u;
    if (__syncthreads_or(!ok)) {
      failed = true;
      break;
    }
    tc::tc_fence_after_sync();
    // ---- epilogue: warp w reads TMEM lanes 32*(w%4).., columns slice w/4
    {
      const int q = warp & 3, j = warp >> 2;
      const int rr = 32 * q + lane;
      const int64_t item = t * kTcRows + rr;
      float* dst = nullptr;
      if (item < nitems) {
        if (MODE == kSegments) {
          const int4 sg = __ldg(segs + item);
          dst = sg.w < 0 ? A + (int64_t)sg.x * L : partial + (int64_t)sg.w * L;
        } else {
          dst = A + item * L;
        }
      }
      constexpr int CW = L / 4;  // columns per warp
#pragma unroll
      for (int c = 0; c < CW; c += 8) {
        float v[8];
        tc::tmem_ld8(tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(j * CW + c), v);
        if (dst != nullptr) {
          float4* o = reinterpret_cast<float4*>(dst + j * CW + c);
          o[0] = make_float4(v[0], v[1], v[2], v[3]);
          o[1] = make_float4(v[4], v[5], v[6], v[7]);
        }
      }
    }
    tc::tc_fence_before_sync();
    __syncthreads();
  }
  if (failed) {
    // the MMAs of the abandoned tile may still be running: wait once more
    // (bounded) before the tensor memory is released
    mbar_wait_timeout(&mbar, phase ^ 1u);
    if (tid == 0) atomicOr(&hdr->error, kErrTimeout);
  }
  tc::tc_fence_before_sync();
  __syncthreads();
  tc::tc_fence_after_sync();
  if (warp == 0) tc::tmem_dealloc(tmem, NCOLS);
}

struct TcLaunch {
  int grid_cap;
  size_t smem;
};

template <int K, int L, int MODE>
cudaError_t tc_setup(TcLaunch* out) {
  static TcLaunch cached[64] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev >= 0 && dev < 64 && cached[dev].grid_cap > 0) {
    *out = cached[dev];
    return cudaSuccess;
  }
  int sm_smem = 0, nsm = 0;
  if ((e = cudaDeviceGetAttribute(&sm_smem, cudaDevAttrMaxSharedMemoryPerMultiprocessor, dev)) != cudaSuccess) return e;
  if ((e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
  size_t smem = tc_smem_bytes(K, L);
  // no more resident CTAs per SM than tensor memory holds accumulators for
  const int max_ctas = 512 / L;
  const size_t floor_bytes = (size_t)sm_smem / (size_t)(max_ctas + 1) + 1;
  if (smem < floor_bytes) smem = floor_bytes;
  if ((e = cudaFuncSetAttribute(k_tc_gemm<K, L, MODE>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem)) !=
      cudaSuccess)
    return e;
  int occ = 0;
  if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, k_tc_gemm<K, L, MODE>, kTcThreads, smem)) !=
      cudaSuccess)
    return e;
  if (occ < 1) return cudaErrorInvalidConfiguration;
  if (occ > max_ctas) occ = max_ctas;
  TcLaunch t{nsm * occ, smem};
  if (dev >= 0 && dev < 64) cached[dev] = t;
  *out = t;
  return cudaSuccess;
}

template <int MODE>
cudaError_t tc_dispatch(int K, int L, int64_t items_upper, WsHeader* hdr, const int4* segs,
                        int max_segs, int64_t dense_rows, const int32_t* crd, const float* vals, const float* X,
                        const float* D, float* A, float* partial, cudaStream_t s) {
#define SLNR_TC_CASE(KK, LL)                                                                              \
  if (K == KK && L == LL) {                                                                               \
    TcLaunch tl;                                                                                          \
    cudaError_t e = tc_setup<KK, LL, MODE>(&tl);                                                          \
    if (e != cudaSuccess) return e;                                                                       \
    int64_t grid = (items_upper + kTcRows - 1) / kTcRows;                                                 \
    if (grid > tl.grid_cap) grid = tl.grid_cap;                                                           \
    if (grid < 1) grid = 1;                                                                               \
    k_tc_gemm<KK, LL, MODE><<<(unsigned)grid, kTcThreads, tl.smem, s>>>(hdr, segs, max_segs,              \
                                                                         dense_rows, crd, vals, X, D, A,  \
                                                                         partial);                        \
    return cudaGetLastError();                                                                            \
  }
  SLNR_TC_CASE(32, 32) SLNR_TC_CASE(32, 64) SLNR_TC_CASE(32, 128) SLNR_TC_CASE(32, 256)
  SLNR_TC_CASE(64, 32) SLNR_TC_CASE(64, 64) SLNR_TC_CASE(64, 128) SLNR_TC_CASE(64, 256)
  SLNR_TC_CASE(128, 32) SLNR_TC_CASE(128, 64) SLNR_TC_CASE(128, 128) SLNR_TC_CASE(128, 256)
#undef SLNR_TC_CASE
  return cudaErrorInvalidValue;
}

}  // namespace

bool tc_supported(int K, int L) {
  return (K == 32 || K == 64 || K == 128) && (L == 32 || L == 64 || L == 128 || L == 256);
}

int seg_scan_blocks(int64_t nrows) { return (int)((nrows + kScanRows - 1) / kScanRows); }

cudaError_t launch_seg_count(const CsrView& B, const SegPlan& plan, cudaStream_t s) {
  if (B.nrows <= 0) return cudaSuccess;
  k_seg_count<<<seg_scan_blocks(B.nrows), kScanThreads, 0, s>>>(B.nrows, B.pos, plan.block_counts);
  return cudaGetLastError();
}

cudaError_t launch_seg_write(const CsrView& B, const SegPlan& plan, cudaStream_t s) {
  if (B.nrows <= 0) return cudaSuccess;
  const int nb = seg_scan_blocks(B.nrows);
  k_seg_write<<<nb, kScanThreads, 0, s>>>(B.nrows, B.pos, plan.block_counts, nb, plan.hdr, plan.segs, plan.heavy,
                                          plan.max_segs, plan.max_heavy, plan.max_chunks);
  return cudaGetLastError();
}

cudaError_t launch_tc_spmm_gemm(int K, int L, const CsrView& B, const float* C, const float* D, float* A,
                                const SegPlan& plan, cudaStream_t s) {
  if (B.nrows <= 0) return cudaSuccess;
  return tc_dispatch<kSegments>(K, L, plan.max_segs, plan.hdr, plan.segs, plan.max_segs, 0, B.crd,
                                B.vals, C, D, A, plan.partial, s);
}

cudaError_t launch_tc_dense_gemm(int64_t M, int K, int L, const float* T, const float* D, float* A,
                                 WsHeader* hdr, cudaStream_t s) {
  if (M <= 0) return cudaSuccess;
  return tc_dispatch<kDense>(K, L, M, hdr, nullptr, 0, M, nullptr, nullptr, T, D, A, nullptr, s);
}

}  // namespace slnr
