// <SpMM,GEMM> / <SpTTM,SpTTM> with the consumer contraction on tcgen05 TF32
// tensor cores.
//
// Fused schedule (Sec. 4.2, Algorithm 1; the temporary is a vector over k,
// Sec. 6.3): for each row r, T(r,:) = sum_p vals[p] C(crd[p],:) is built on
// chip and A(r,:) = T(r,:) . D follows at once.  Rows are grouped into
// "segments" of at most kSegChunk nonzeros (a row with more nonzeros becomes
// several chunk segments); a persistent CTA takes 128 segments at a time:
//   producer: 27 warps gather C rows into registers and write the 128 x K
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
// variant) by D: the producer reads T rows instead of gathering them.  In
// Hadamard mode (<SpMMH,GEMM>) the gathered row is C(k,:) .* C2(k,:).
#include "launch.h"
#include "tcgen05.cuh"

namespace slnr {

namespace {

constexpr int kTcThreads = 1024;
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

// Waits until *count >= target (a monotonic shared-memory counter); false on timeout.
__device__ __forceinline__ bool count_wait_timeout(const int* count, int target) {
  const long long t0 = clock64();
  while (tc::ld_acquire_smem(count) < target) {
    __nanosleep(64);  // leave the issue slots to the warps that are working
    if (clock64() - t0 > kWaitCycles) return false;
  }
  return true;
}

#ifndef SLNR_TC_MBAR_SLEEP
#define SLNR_TC_MBAR_SLEEP 256  // back-off (ns) between polls of an mbarrier by the MMA and epilogue warps
#endif

// Waits for the phase with the given parity to complete; false on timeout.
// Sleeps between polls so that the waiting MMA and epilogue warps leave the
// issue slots to the producers (their work has slack of a whole tile).
__device__ __forceinline__ bool mbar_wait_timeout(uint64_t* bar, uint32_t parity) {
  const long long t0 = clock64();
  while (!tc::mbar_try_wait(bar, parity)) {
    if (SLNR_TC_MBAR_SLEEP > 0) __nanosleep(SLNR_TC_MBAR_SLEEP);
    if (clock64() - t0 > kWaitCycles) return false;
  }
  return true;
}

// Waits for the phase with the given parity to complete (1), or until
// *end <= j, i.e. there is no tile j to wait for (0); -1 on timeout.
__device__ __forceinline__ int mbar_wait_or_end(uint64_t* bar, uint32_t parity, const int* end, int j) {
  const long long t0 = clock64();
  while (!tc::mbar_try_wait(bar, parity)) {
    if (*reinterpret_cast<const volatile int*>(end) <= j) return 0;
    if (SLNR_TC_MBAR_SLEEP > 0) __nanosleep(SLNR_TC_MBAR_SLEEP);
    if (clock64() - t0 > kWaitCycles) return -1;
  }
  return 1;
}

// kSegments: gathered row segments; kSegmentsH: the same with Hadamard rows
// X[k,:] .* X2[k,:] (<SpMMH,GEMM>); kDense: rows of a materialised T.
enum TcMode { kSegments = 0, kDense = 1, kSegmentsH = 2 };

// Columns of the T tile and of D^T: K, padded to one 128-byte swizzle atom
// (32 tf32 values) when K = 16; the padding columns hold zeros.
__host__ __device__ constexpr int tc_kt(int K) { return K < 32 ? 32 : K; }

// Number of T / accumulator buffers: up to four, as many as fit beside D^T
// in shared memory (200 KB budget) and in tensor memory (512 columns).
__host__ __device__ constexpr int tc_nbuf(int K, int L) {
  return ((size_t)4 * kTcRows * tc_kt(K) * 4 + (size_t)L * tc_kt(K) * 4 + 1024 <= (size_t)200 * 1024 && 4 * L <= 512)
             ? 4
             : ((size_t)2 * kTcRows * tc_kt(K) * 4 + (size_t)L * tc_kt(K) * 4 + 1024 <= (size_t)200 * 1024 &&
                2 * L <= 512)
                   ? 2
                   : 1;
}

// Shared memory: NBUF T tiles (kTcRows x KT) and D^T (L x KT), tf32 K-major
// 128B-swizzled, plus 1 KB of alignment slack.
__host__ __device__ constexpr size_t tc_smem_bytes(int K, int L) {
  return (size_t)tc_nbuf(K, L) * kTcRows * tc_kt(K) * 4 + (size_t)L * tc_kt(K) * 4 + 1024;
}

#ifndef SLNR_TC_VPL
#define SLNR_TC_VPL 4  // T-row columns per producer lane (4, 8 or 16)
#endif
#ifndef SLNR_TC_UNROLL
#define SLNR_TC_UNROLL 8  // gathered rows in flight per lane group
#endif
#ifndef SLNR_TC_DENSE_ROWS
#define SLNR_TC_DENSE_ROWS 4  // DENSE mode: rows of T loaded at once per lane group
#endif

// Producer layout: a T row is built by a group of GS = K / VPL lanes, lane gl
// of the group holding the VPL columns [VPL*gl, VPL*gl + VPL), loaded as
// float4s; a warp builds G = 32 / GS rows at once, one per group, with U row
// gathers in flight per group.  A claim is the G consecutive items of one
// warp pass.
#ifndef SLNR_TC_TAIL_BATCH
#define SLNR_TC_TAIL_BATCH 1  // segments without prefetch: the last batch loaded at once (0: row by row)
#endif
#ifndef SLNR_TC_SEQ_SEGS
#define SLNR_TC_SEQ_SEGS 2  // segments a lane group claims at once and gathers one after the other
#endif
#ifndef SLNR_TC_PF_AHEAD
#define SLNR_TC_PF_AHEAD 8  // rows of a segment prefetched into L2 beyond the batch in flight
#endif

// L2 prefetch of the 128-byte line holding p (no register, nothing to wait for).
__device__ __forceinline__ void prefetch_line(const void* p) { asm volatile("prefetch.global.L2 [%0];" ::"l"(p)); }

// acc += sum_{p in [p0,p1)} vals[p] * R(crd[p])[col .. col+VPL), sequential in p,
// where R(k) = X[k,:] (or X[k,:] .* X2[k,:] with H).  U rows are loaded per
// batch (the last batch predicated, so a short segment costs one round trip
// per batch, not per row).  Rows further ahead are pulled into L2 by line
// prefetches, which hold no register: each of the group's GS lanes prefetches
// one 128-byte line, RPI = GS / LPR rows per step, and the front is kept AHEAD
// rows beyond the batch in flight.
template <int K, int VPL, int U, int AHEAD, bool H>
__device__ __forceinline__ void gather_pf(float (&acc)[VPL], const int32_t* __restrict__ crd,
                                          const float* __restrict__ vals, int p0, int p1,
                                          const float* __restrict__ X, const float* __restrict__ X2, int col,
                                          int gl) {
  constexpr int GS = K / VPL, LPR = K >= 32 ? K / 32 : 1, RPI = GS / LPR;  // a row of 16 floats is half a line
  static_assert(AHEAD % RPI == 0, "the prefetch window is whole steps");
  constexpr int NPF = AHEAD / RPI;
  const int prow = gl / LPR, poff = (gl % LPR) * 32;
  auto pf_row = [&](int c) {
    prefetch_line(X + (int64_t)c * K + poff);
    if constexpr (H) prefetch_line(X2 + (int64_t)c * K + poff);
  };
  int pq = p0 + U;  // first row not covered by the first batch or the window
  int pf = -1;      // coordinate of row pq + prow (the next prefetch step)
  if constexpr (NPF > 0) {
    int cs[NPF];
#pragma unroll
    for (int k = 0; k < NPF; ++k) {
      const int q = pq + k * RPI + prow;
      cs[k] = q < p1 ? __ldg(crd + q) : -1;
    }
    pq += AHEAD;
    pf = pq + prow < p1 ? __ldg(crd + pq + prow) : -1;
#pragma unroll
    for (int k = 0; k < NPF; ++k)
      if (cs[k] >= 0) pf_row(cs[k]);
  }
  // advances the prefetch front by one step when it is within AHEAD rows of p + U
  auto advance = [&](int p) {
    if constexpr (NPF > 0) {
      if (pq < p + U + AHEAD && pq < p1) {
        if (pf >= 0) pf_row(pf);
        pq += RPI;
        pf = pq + prow < p1 ? __ldg(crd + pq + prow) : -1;
      }
    }
  };
  auto row = [&](float (&x)[VPL], int c) {
    ldg_vec<VPL>(x, X + (int64_t)c * K + col);
    if constexpr (H) {
      float x2[VPL];
      ldg_vec<VPL>(x2, X2 + (int64_t)c * K + col);
#pragma unroll
      for (int e = 0; e < VPL; ++e) x[e] *= x2[e];
    }
  };
  int p = p0;
  for (; p + U <= p1; p += U) {  // full batches
    advance(p);
    int c[U];
    float v[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      c[u] = __ldg(crd + p + u);
      v[u] = __ldg(vals + p + u);
    }
    float x[U][VPL];
#pragma unroll
    for (int u = 0; u < U; ++u) row(x[u], c[u]);
#pragma unroll
    for (int u = 0; u < U; ++u)
#pragma unroll
      for (int e = 0; e < VPL; ++e) acc[e] = fmaf(v[u], x[u][e], acc[e]);
  }
  if (p < p1) {  // the last, partial batch (all its loads still in flight together)
    advance(p);
    int c[U];
    float v[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const bool ok = p + u < p1;
      c[u] = ok ? __ldg(crd + p + u) : -1;
      v[u] = ok ? __ldg(vals + p + u) : 0.f;
    }
    float x[U][VPL];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      if (c[u] >= 0) row(x[u], c[u]); else zero_vec(x[u]);
    }
#pragma unroll
    for (int u = 0; u < U; ++u)
      if (c[u] >= 0)
#pragma unroll
        for (int e = 0; e < VPL; ++e) acc[e] = fmaf(v[u], x[u][e], acc[e]);
  }
}

template <int K>
struct ProdLayout {
  static constexpr int VPL = K / SLNR_TC_VPL >= 1 && K / SLNR_TC_VPL <= 32 ? SLNR_TC_VPL : 4;
  static constexpr int GS = K / VPL;
  static constexpr int G = 32 / GS;
  static constexpr int U = SLNR_TC_UNROLL;
  static_assert(VPL == 4 || VPL == 8 || VPL == 16, "VPL must be 4, 8 or 16");
  static_assert(GS >= 1 && GS <= 32 && 32 % GS == 0, "a group is a power-of-two part of a warp");
};

// Stores the VPL values of lane group column col of T row s (buffer sTb),
// rounded to tf32, into the 128B-swizzled K-major tile.
template <int VPL>
__device__ __forceinline__ void store_t_part(uint8_t* sTb, int s, int col, const float (&acc)[VPL]) {
#pragma unroll
  for (int h = 0; h < VPL / 4; ++h)
    *reinterpret_cast<uint4*>(sTb + tc::sw128_offset(s, col + 4 * h, kTcRows)) =
        make_uint4(tc::to_tf32(acc[4 * h]), tc::to_tf32(acc[4 * h + 1]), tc::to_tf32(acc[4 * h + 2]),
                   tc::to_tf32(acc[4 * h + 3]));
}

// Warp roles of the persistent tile kernel (32 warps):
//   warps 0..26  producers: claim G consecutive items of this CTA's item
//                tiles at a time (in order), build their T rows with one lane
//                group per row, and store each row into its item's slot of
//                the tile's T buffer with its destination; one mbarrier
//                arrival per claim;
//   warp 27      MMA issuer: waits full[b] (every claim of the tile placed)
//                and free[b] (buffer's previous accumulator drained), issues
//                the tile's K/8 tcgen05.mma into TMEM accumulator b, commits
//                to mma[b];
//   warps 28..31 epilogue: wait mma[b], read TMEM lane quadrant (warp % 4),
//                write A rows or partial rows, arrive free[b].
// Item tile n uses buffer n % NBUF; a producer stores into it only after the
// MMAs of tile n - NBUF completed.  Claims are taken in order, so the claim a
// producer waits on belongs to an earlier tile, which only needs earlier
// claims (no cycle).  Producers wait on mma_tiles_done, a monotonic count of
// completed tiles that the epilogue publishes (release) once all four
// epilogue warps have read the tile's row destinations.  Every wait is
// bounded; a timeout raises kErrTimeout and the CTA winds down.
// Items per producer claim: SLNR_TC_SEQ_SEGS segments per lane group, or
// SLNR_TC_DENSE_ROWS rows per lane group in DENSE mode.
template <int K, int MODE>
__host__ __device__ constexpr int claim_items() {
  return ProdLayout<K>::G * (MODE == kDense ? SLNR_TC_DENSE_ROWS : SLNR_TC_SEQ_SEGS);
}

constexpr int kProducerWarps = 27;
constexpr int kTileRing = 16;  // local tiles whose global index is kept in shared memory
constexpr int kMmaWarp = 27;  // warps 28..31: epilogue

template <int K, int L, int MODE, bool PF>
__global__ void __launch_bounds__(kTcThreads, 1)
    k_tc_gemm(WsHeader* hdr, const int4* __restrict__ segs, int max_segs,
              int64_t dense_rows, const int32_t* __restrict__ crd, const float* __restrict__ vals,
              const float* __restrict__ X, const float* __restrict__ X2, const float* __restrict__ D,
              float* __restrict__ A,
              float* __restrict__ partial) {
  static_assert(K == 16 || K == 32 || K == 64 || K == 128, "K must be 16, 32, 64 or 128");
  static_assert(L % 16 == 0 && L >= 16 && L <= 256, "L must be a multiple of 16 in [16, 256]");
  constexpr int KT = tc_kt(K);  // tile columns (K, or 32 with zero padding)
  static_assert(kTcThreads == 1024, "32 warps: 27 producers, 1 MMA, 4 epilogue");
  using PL = ProdLayout<K>;
  constexpr int NBUF = tc_nbuf(K, L);
  constexpr uint32_t IDESC = tc::idesc_tf32(kTcRows, L);
  constexpr uint32_t NCOLS = NBUF * L;  // TMEM columns: NBUF fp32 accumulators
  constexpr int TBYTES = kTcRows * KT * 4;
  extern __shared__ uint8_t smem_raw[];
  __shared__ uint64_t full_bar[NBUF], mma_bar[NBUF], free_bar[NBUF];
  __shared__ int2 dest[NBUF][kTcRows];  // per slot: (A row, partial slot); x < 0 = padding
  __shared__ uint32_t tmem_base;
  __shared__ int claim, fill, fail_flag, mma_tiles_done;
  __shared__ int tile_gid[kTileRing], tile_seq[kTileRing], end_tile;
  __shared__ int last_commit[NBUF];     // last tile committed to each accumulator (-1: none)
  uint8_t* sT = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sD = sT + NBUF * TBYTES;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (warp == kMmaWarp) {
    tc::tmem_alloc(&tmem_base, NCOLS);
    tc::tmem_relinquish();
  }
  if (tid == 0) {
    for (int b = 0; b < NBUF; ++b) {
      tc::mbar_init(&full_bar[b], kTcRows / claim_items<K, MODE>());  // one arrival per claim
      tc::mbar_init(&mma_bar[b], 1);
      tc::mbar_init(&free_bar[b], 4);
      last_commit[b] = -1;
    }
    tc::fence_mbar_init();
    claim = 0;
    fill = 0;
    fail_flag = 0;
    mma_tiles_done = 0;
  }
  // Item tiles are handed out dynamically: CTAs take them from a global
  // counter in the workspace header (zeroed before the launch), one tile
  // ahead of need, so the hub rows' costly tiles do not pile up on a few SMs.
  // Local tile j's global index is published in a small shared ring
  // (tile_gid, with tile_seq = j + 1 once written); the first local tile
  // whose index lies past the last item tile is end_tile, and every role
  // stops there.
  int64_t nitems;
  if (MODE != kDense) {
    const int n = hdr->n_segs;
    nitems = n < max_segs ? n : max_segs;
  } else {
    nitems = dense_rows;
  }
  const int64_t ntiles = (nitems + kTcRows - 1) / kTcRows;
  if (tid == 0) {
    for (int r = 0; r < kTileRing; ++r) tile_seq[r] = 0;
    const int g0 = atomicAdd(&hdr->next_tile, 1);
    tile_gid[0] = g0;
    tile_seq[0] = 1;
    end_tile = g0 >= ntiles ? 0 : INT_MAX;
  }
  // D (K x L, row-major) -> D^T as the B operand (L rows of KT), tf32; rows
  // k >= K of the padded tile are zero
  for (int i = tid; i < KT * (L / 4); i += kTcThreads) {
    const int k = i / (L / 4), n4 = i % (L / 4);
    const float4 d = k < K ? __ldg(reinterpret_cast<const float4*>(D + (int64_t)k * L) + n4)
                           : make_float4(0.f, 0.f, 0.f, 0.f);
    const float dv[4] = {d.x, d.y, d.z, d.w};
#pragma unroll
    for (int e = 0; e < 4; ++e)
      *reinterpret_cast<uint32_t*>(sD + tc::sw128_offset(4 * n4 + e, k, L)) = tc::to_tf32(dv[e]);
  }
  if constexpr (KT > K) {  // the padding columns of every T buffer: zero once, never written
    for (int i = tid; i < NBUF * kTcRows * (KT - K); i += kTcThreads) {
      const int b = i / (kTcRows * (KT - K)), r = (i / (KT - K)) % kTcRows, k = K + i % (KT - K);
      *reinterpret_cast<uint32_t*>(sT + b * TBYTES + tc::sw128_offset(r, k, kTcRows)) = 0u;
    }
  }
  tc::fence_proxy_async_smem();
  tc::tc_fence_before_sync();
  __syncthreads();
  tc::tc_fence_after_sync();
  const uint32_t tmem = tmem_base;

  // global item tile of local tile t: >= 0 once known, -1 if t does not
  // exist (t >= end_tile), -2 if the wait timed out
  auto tile_of = [&](int t) -> int {
    const long long t0 = clock64();
    while (tc::ld_acquire_smem(&tile_seq[t % kTileRing]) != t + 1) {
      if (*reinterpret_cast<volatile int*>(&end_tile) <= t) return -1;
      __nanosleep(32);
      if (clock64() - t0 > kWaitCycles) return -2;
    }
    const int gid = *reinterpret_cast<volatile int*>(&tile_gid[t % kTileRing]);
    return gid < ntiles ? gid : -1;
  };
  // the first claim of local tile t fetches the global index of tile t + 1
  auto fetch_next_tile = [&](int t) {
    const int gnext = atomicAdd(&hdr->next_tile, 1);
    tile_gid[(t + 1) % kTileRing] = gnext;
    if (gnext >= ntiles) atomicMin(&end_tile, t + 1);
    tc::st_release_smem(&tile_seq[(t + 1) % kTileRing], t + 2);
  };

  if (warp < kProducerWarps) {
    // ---------------- producers ----------------
    // A claim covers IPC = G * R consecutive items of local item tile c / CPT:
    // lane group g builds the T rows of items g, g + G, ..., g + (R-1) G of
    // the claim (R = 1 gathered segment, or R = U rows of a materialised T in
    // DENSE mode, all loads in flight at once).  It builds the rows first,
    // then waits for its buffer to be free (the MMAs of tile c / CPT - NBUF
    // completed and their destinations read), stores the rows and their
    // destinations, and lane 0 arrives once for the claim.
    constexpr int VPL = PL::VPL, G = PL::G, R = MODE != kDense ? SLNR_TC_SEQ_SEGS : SLNR_TC_DENSE_ROWS;
    constexpr int IPC = G * R, CPT = kTcRows / IPC;
    static_assert(IPC == claim_items<K, MODE>(), "barrier count matches the claims");
    static_assert(kTcRows % IPC == 0, "claims tile the item tile");
    const int g = lane / PL::GS, col = (lane % PL::GS) * VPL;
    // record of item g + r G of claim c, whose item tile has global index gid
    auto load_rec = [&](int gid, int c, int r) -> int4 {
      int4 rv = make_int4(-1, 0, 0, -1);
      const int64_t item = (int64_t)gid * kTcRows + (c % CPT) * IPC + r * G + g;
      if (item < nitems) rv = (MODE != kDense) ? __ldg(segs + item) : make_int4((int)item, 0, 0, -1);
      return rv;
    };
    // takes the next claim of this CTA; returns its item tile's global index
    // (< 0: no such tile / timeout).  The first claim of a local tile also
    // fetches the next local tile's global index.
    int known_tile = -1, known_gid = -1;  // the last local tile this warp resolved
    auto take_claim = [&](int& c) -> int {
      int v = 0;
      if (lane == 0) v = atomicAdd(&claim, 1);
      c = __shfl_sync(0xffffffffu, v, 0);
      const int t = c / CPT;
      if (t != known_tile) {
        known_gid = __shfl_sync(0xffffffffu, tile_of(t), 0);
        known_tile = known_gid >= 0 ? t : -1;
      }
      const int gid = known_gid;
      if (gid >= 0 && c % CPT == 0) {
        if (lane == 0) fetch_next_tile(t);
        __syncwarp();
      }
      return gid;
    };
    int cl = 0;
    int gid = take_claim(cl);
    int4 rec = gid >= 0 ? load_rec(gid, cl, 0) : make_int4(-1, 0, 0, -1);  // segment record (R = 1)
    while (gid >= 0) {
      int cl_next = 0;
      const int gid_next = take_claim(cl_next);
      float acc[R][VPL];
      int2 dst0 = make_int2(-1, -1);  // destination of the segment (R = 1)
      if constexpr (MODE != kDense) {
        // the group's R segments, one after the other (the first record was
        // loaded with the previous claim; the others share its cache line)
        int4 rr[R];
        rr[0] = rec;
#pragma unroll
        for (int r = 1; r < R; ++r) rr[r] = load_rec(gid, cl, r);
        const int4 rec_next = gid_next >= 0 ? load_rec(gid_next, cl_next, 0) : make_int4(-1, 0, 0, -1);
        constexpr bool H = MODE == kSegmentsH;
        constexpr int UG = H ? PL::U / 2 : PL::U;  // two loads per nonzero in Hadamard mode
#pragma unroll
        for (int r = 0; r < R; ++r) {
          zero_vec(acc[r]);
          if (rr[r].x >= 0) {
            if constexpr (PF)
              gather_pf<K, VPL, UG, SLNR_TC_PF_AHEAD, H>(acc[r], crd, vals, rr[r].y, rr[r].z, X, X2, col,
                                                          lane % PL::GS);
            else if constexpr (SLNR_TC_TAIL_BATCH)
              gather_pf<K, VPL, UG, 0, H>(acc[r], crd, vals, rr[r].y, rr[r].z, X, X2, col, lane % PL::GS);
            else
              gather_acc<VPL, UG, H>(acc[r], crd, vals, rr[r].y, rr[r].z, X, K, col, X2);
          }
        }
        dst0 = make_int2(rr[0].x, rr[0].w);
        rec = rec_next;
      } else {
#pragma unroll
        for (int r = 0; r < R; ++r) {
          const int4 rr = load_rec(gid, cl, r);
          if (rr.x >= 0) ldg_vec<VPL>(acc[r], X + (int64_t)rr.x * K + col); else zero_vec(acc[r]);
        }
      }
      __syncwarp();
      // the claim's IPC rows take the next IPC slots in completion order, so a
      // long segment delays only its own rows, never a whole tile (the item
      // tiles of this CTA, and the slot tiles the MMAs consume, are as many)
      int sl = 0;
      if (lane == 0) sl = atomicAdd(&fill, IPC);
      sl = __shfl_sync(0xffffffffu, sl, 0);
      const int j = sl / kTcRows, b = j % NBUF, s0 = sl % kTcRows + g;
      if (j >= NBUF) {
        const bool ok = count_wait_timeout(&mma_tiles_done, j - NBUF + 1);
        if (!__all_sync(0xffffffffu, ok)) {
          atomicOr(&fail_flag, 1);
          break;
        }
      }
#pragma unroll
      for (int r = 0; r < R; ++r) {
        store_t_part<VPL>(sT + b * TBYTES, s0 + r * G, col, acc[r]);
        if (lane % PL::GS == 0) {
          if constexpr (MODE == kDense) {
            dest[b][s0 + r * G] = make_int2(load_rec(gid, cl, r).x, -1);
          } else if (r == 0) {
            dest[b][s0] = dst0;
          } else {
            const int4 rq = load_rec(gid, cl, r);
            dest[b][s0 + r * G] = make_int2(rq.x, rq.w);
          }
        }
      }
      tc::fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&full_bar[b]);
      if (gid_next == -2) {  // timed out waiting for a tile index
        atomicOr(&fail_flag, 1);
        break;
      }
      cl = cl_next;
      gid = gid_next;
    }
    if (gid == -2) atomicOr(&fail_flag, 1);
  } else if (warp == kMmaWarp) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      const uint32_t sT_addr = tc::smem_u32(sT), sD_addr = tc::smem_u32(sD);
      for (int j = 0;; ++j) {
        const int b = j % NBUF;
        const int st = mbar_wait_or_end(&full_bar[b], (j / NBUF) & 1, &end_tile, j);
        if (st == 0) break;  // this CTA has no tile j
        if (st < 0 || (j >= NBUF && !mbar_wait_timeout(&free_bar[b], ((j / NBUF) - 1) & 1))) {
          atomicOr(&fail_flag, 1);
          break;
        }
        tc::tc_fence_after_sync();
        const uint32_t a_base = sT_addr + b * TBYTES;
#pragma unroll
        for (int kb = 0; kb < KT / 32; ++kb)
#pragma unroll
          for (int ks = 0; ks < 4; ++ks) {
            const uint64_t ad = tc::desc_k_sw128(a_base + kb * kTcRows * 128 + ks * 32);
            const uint64_t bd = tc::desc_k_sw128(sD_addr + kb * L * 128 + ks * 32);
            tc::mma_tf32(tmem + (uint32_t)(b * L), ad, bd, IDESC, (kb | ks) != 0);
          }
        tc::mma_commit(&mma_bar[b]);
        last_commit[b] = j;
      }
    }
    __syncwarp();
  } else {
    // ---------------- epilogue ----------------
    const int q = warp & 3;  // TMEM lane quadrant of this warp
    for (int j = 0;; ++j) {
      const int b = j % NBUF;
      const int st = __shfl_sync(0xffffffffu, mbar_wait_or_end(&mma_bar[b], (j / NBUF) & 1, &end_tile, j), 0);
      if (st == 0) break;  // this CTA has no tile j
      if (st < 0) {
        atomicOr(&fail_flag, 1);
        break;
      }
      tc::tc_fence_after_sync();
      const int rr = 32 * q + lane;
      const int2 dd = dest[b][rr];
      // all four epilogue warps have their destinations: the slot tile may be refilled
      asm volatile("bar.sync 1, 128;" ::: "memory");
      if (q == 0 && lane == 0) tc::st_release_smem(&mma_tiles_done, j + 1);
      float* dst = nullptr;
      if (dd.x >= 0) dst = dd.y < 0 ? A + (int64_t)dd.x * L : partial + (int64_t)dd.y * L;
      if constexpr (L >= 32) {
#pragma unroll 1
        for (int c = 0; c < L; c += 32) {
          float v[32];
          tc::tmem_ld32(tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(b * L + c), v);
          if (dst != nullptr) {
            float4* o = reinterpret_cast<float4*>(dst + c);
#pragma unroll
            for (int i = 0; i < 8; ++i) o[i] = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
          }
        }
      } else {
        float v[16];
        tc::tmem_ld16(tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(b * L), v);
        if (dst != nullptr) {
          float4* o = reinterpret_cast<float4*>(dst);
#pragma unroll
          for (int i = 0; i < 4; ++i) o[i] = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
        }
      }
      tc::tc_fence_before_sync();
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&free_bar[b]);
    }
  }

  // ---- teardown: every role has finished its loop
  tc::tc_fence_before_sync();
  __syncthreads();
  if (fail_flag) {
    // MMAs of abandoned tiles may still be running: wait (bounded) for each
    // accumulator's last commit before the tensor memory is released
    if (warp == kMmaWarp && lane == 0)
      for (int b = 0; b < NBUF; ++b)
        if (last_commit[b] >= 0) mbar_wait_timeout(&mma_bar[b], (last_commit[b] / NBUF) & 1);
    if (tid == 0) atomicOr(&hdr->error, kErrTimeout);
  }
  __syncthreads();
  tc::tc_fence_after_sync();
  if (warp == kMmaWarp) tc::tmem_dealloc(tmem, NCOLS);
}

struct TcLaunch {
  int grid_cap;
  size_t smem;
};

template <int K, int L, int MODE, bool PF>
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
  // no more resident CTAs per SM than tensor memory (512 columns) holds
  // accumulators for: a CTA waiting in tcgen05.alloc would only idle
  const int max_ctas = 512 / (tc_nbuf(K, L) * L);
  const size_t floor_bytes = (size_t)sm_smem / (size_t)(max_ctas + 1) + 1;
  if (smem < floor_bytes) smem = floor_bytes;
  if ((e = cudaFuncSetAttribute(k_tc_gemm<K, L, MODE, PF>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem)) !=
      cudaSuccess)
    return e;
  if ((e = cudaFuncSetAttribute(k_tc_gemm<K, L, MODE, PF>, cudaFuncAttributePreferredSharedMemoryCarveout,
                                (int)cudaSharedmemCarveoutMaxShared)) != cudaSuccess)
    return e;
  int occ = 0;
  if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, k_tc_gemm<K, L, MODE, PF>, kTcThreads, smem)) !=
      cudaSuccess)
    return e;
  if (occ < 1) return cudaErrorInvalidConfiguration;
  if (occ > max_ctas) occ = max_ctas;
  TcLaunch t{nsm * occ, smem};
  if (dev >= 0 && dev < 64) cached[dev] = t;
  *out = t;
  return cudaSuccess;
}

template <int MODE, bool PF>
cudaError_t tc_dispatch(int K, int L, int64_t items_upper, WsHeader* hdr, const int4* segs,
                        int max_segs, int64_t dense_rows, const int32_t* crd, const float* vals, const float* X,
                        const float* X2, const float* D, float* A, float* partial, cudaStream_t s) {
#define SLNR_TC_CASE(KK, LL)                                                                              \
  if (K == KK && L == LL) {                                                                               \
    TcLaunch tl;                                                                                          \
    cudaError_t e = tc_setup<KK, LL, MODE, PF>(&tl);                                                      \
    if (e != cudaSuccess) return e;                                                                       \
    int64_t grid = (items_upper + kTcRows - 1) / kTcRows;                                                 \
    if (grid > tl.grid_cap) grid = tl.grid_cap;                                                           \
    if (grid < 1) grid = 1;                                                                               \
    if ((e = cudaMemsetAsync(&hdr->next_tile, 0, sizeof(int), s)) != cudaSuccess) return e;               \
    k_tc_gemm<KK, LL, MODE, PF><<<(unsigned)grid, kTcThreads, tl.smem, s>>>(hdr, segs, max_segs,          \
                                                                             dense_rows, crd, vals, X,    \
                                                                             X2, D, A, partial);          \
    return cudaGetLastError();                                                                            \
  }
  SLNR_TC_CASE(16, 16) SLNR_TC_CASE(16, 32) SLNR_TC_CASE(16, 64) SLNR_TC_CASE(16, 128) SLNR_TC_CASE(16, 256)
  SLNR_TC_CASE(32, 16) SLNR_TC_CASE(32, 32) SLNR_TC_CASE(32, 64) SLNR_TC_CASE(32, 128) SLNR_TC_CASE(32, 256)
  SLNR_TC_CASE(64, 16) SLNR_TC_CASE(64, 32) SLNR_TC_CASE(64, 64) SLNR_TC_CASE(64, 128) SLNR_TC_CASE(64, 256)
  SLNR_TC_CASE(128, 16) SLNR_TC_CASE(128, 32) SLNR_TC_CASE(128, 64) SLNR_TC_CASE(128, 128) SLNR_TC_CASE(128, 256)
#undef SLNR_TC_CASE
  return cudaErrorInvalidValue;
}

// L2 size of the current device (cached per device; 0 if it cannot be read).
size_t l2_bytes() {
  static size_t cached[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  if (cached[dev] == 0) {
    int v = 0;
    if (cudaDeviceGetAttribute(&v, cudaDevAttrL2CacheSize, dev) != cudaSuccess) return 0;
    cached[dev] = (size_t)v;
  }
  return cached[dev];
}

}  // namespace

bool tc_supported(int K, int L) {
  return (K == 16 || K == 32 || K == 64 || K == 128) && (L == 16 || L == 32 || L == 64 || L == 128 || L == 256) &&
         tc_smem_bytes(K, L) <= (size_t)200 * 1024;
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
                                const SegPlan& plan, cudaStream_t s, const float* C2) {
  if (B.nrows <= 0) return cudaSuccess;
  // Gathered rows that do not fit in half of L2 miss often: the producers
  // then prefetch the rows ahead of their gathers into L2 (gather_pf).
  const bool pf = (size_t)B.ncols * (size_t)K * sizeof(float) * (C2 != nullptr ? 2 : 1) > l2_bytes() / 2;
  if (C2 != nullptr)
    return pf ? tc_dispatch<kSegmentsH, true>(K, L, plan.max_segs, plan.hdr, plan.segs, plan.max_segs, 0, B.crd,
                                              B.vals, C, C2, D, A, plan.partial, s)
              : tc_dispatch<kSegmentsH, false>(K, L, plan.max_segs, plan.hdr, plan.segs, plan.max_segs, 0, B.crd,
                                               B.vals, C, C2, D, A, plan.partial, s);
  return pf ? tc_dispatch<kSegments, true>(K, L, plan.max_segs, plan.hdr, plan.segs, plan.max_segs, 0, B.crd,
                                           B.vals, C, nullptr, D, A, plan.partial, s)
            : tc_dispatch<kSegments, false>(K, L, plan.max_segs, plan.hdr, plan.segs, plan.max_segs, 0, B.crd,
                                            B.vals, C, nullptr, D, A, plan.partial, s);
}

cudaError_t launch_tc_dense_gemm(int64_t M, int K, int L, const float* T, const float* D, float* A,
                                 WsHeader* hdr, cudaStream_t s) {
  if (M <= 0) return cudaSuccess;
  return tc_dispatch<kDense, false>(K, L, M, hdr, nullptr, 0, M, nullptr, nullptr, T, nullptr, D, A, nullptr, s);
}

}  // namespace slnr
