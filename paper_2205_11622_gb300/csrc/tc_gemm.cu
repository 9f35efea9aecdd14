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

#ifndef SLNR_TC_WARPS
#define SLNR_TC_WARPS 32  // warps of the tile kernel's CTA: producers, then one MMA warp, then four epilogue warps
#endif
constexpr int kTcWarps = SLNR_TC_WARPS;
constexpr int kTcThreads = 32 * kTcWarps;
static_assert(kTcWarps % 4 == 0 && kTcWarps >= 8, "the four epilogue warps are a whole warpgroup");
constexpr int kTcRows = 128;  // MMA M
constexpr int kScanRows = 2048;
constexpr int kScanThreads = 256;
constexpr int kRowsPerThread = kScanRows / kScanThreads;

__device__ __forceinline__ int segs_of(int n) { return n <= kSegChunk ? 1 : (n + kSegChunk - 1) / kSegChunk; }

// Segments are listed by length class, longest first, so that the items a
// lane group takes together have similar lengths and one batch shape fits
// them all (a short segment would otherwise pay for a whole predicated batch
// of row loads).  Class of a segment of n nonzeros: n in (64,128] -> 0,
// (32,64] -> 1, ..., 2 -> 6, 1 -> 7, empty -> 8.  Long segments first also
// keeps the costly item tiles away from the end of the kernel.
__device__ __forceinline__ int seg_class(int n) {
  const int c = n <= 1 ? 0 : 32 - __clz(n - 1);  // ceil(log2(n)) for n >= 1
  return n == 0 ? kSegClasses - 1 : kSegClasses - 2 - c;
}

// Inclusive block scan of N ints (kScanThreads threads); returns the block
// totals in tot.
template <int N>
__device__ __forceinline__ void block_scan(int (&v)[N], int (&tot)[N]) {
  __shared__ int wsum[kScanThreads / 32][N];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int q = 0; q < N; ++q)
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, v[q], o);
      if (lane >= o) v[q] += y;
    }
  if (lane == 31)
#pragma unroll
    for (int q = 0; q < N; ++q) wsum[warp][q] = v[q];
  __syncthreads();
#pragma unroll
  for (int q = 0; q < N; ++q) {
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

// Adds one row of n nonzeros to the counters: segments per class
// (kSegClasses of them), then heavy rows, then chunks of heavy rows.
__device__ __forceinline__ void count_row(int n, int (&v)[kSegCounters]) {
  const int ns = segs_of(n);
  const int q = seg_class(ns == 1 ? n : n - (ns - 1) * kSegChunk);  // the row's (last) segment
#pragma unroll
  for (int k = 0; k < kSegClasses; ++k) v[k] += (k == q) + (k == 0 ? ns - 1 : 0);  // full chunks: class 0
  v[kSegClasses] += ns > 1;
  v[kSegClasses + 1] += ns > 1 ? ns : 0;
}

// Pass 1: the counters of each block of kScanRows rows.
__global__ void __launch_bounds__(kScanThreads) k_seg_count(int nrows, const int32_t* __restrict__ pos,
                                                            int* __restrict__ counts) {
  const int64_t r0 = (int64_t)blockIdx.x * kScanRows + (int64_t)threadIdx.x * kRowsPerThread;
  int v[kSegCounters] = {};
  for (int i = 0; i < kRowsPerThread; ++i) {
    const int64_t r = r0 + i;
    if (r < nrows) count_row(pos[r + 1] - pos[r], v);
  }
  int tot[kSegCounters];
  block_scan<kSegCounters>(v, tot);
  if (threadIdx.x < kSegCounters) counts[kSegCounters * blockIdx.x + threadIdx.x] = tot[threadIdx.x];
}

// Pass 2: each block adds up the counters of all blocks (the class sizes) and
// of the blocks before it, scans its rows and writes their segments into
// their classes' ranges (row order within a class), the heavy-row records
// and the chunk slots (row order).  No atomic decides a position, so the
// lists are the same on every run.  Block 0 publishes the totals in the
// workspace header.
__global__ void __launch_bounds__(kScanThreads) k_seg_write(int nrows, const int32_t* __restrict__ pos,
                                                            const int* __restrict__ counts, int nblocks,
                                                            WsHeader* hdr, int4* __restrict__ segs,
                                                            HeavyRow* __restrict__ heavy, int max_segs,
                                                            int max_heavy, int max_chunks) {
  __shared__ int pre_s[kSegCounters], all_s[kSegCounters];
  if (threadIdx.x < kSegCounters) pre_s[threadIdx.x] = all_s[threadIdx.x] = 0;
  __syncthreads();
  {
    int pre[kSegCounters] = {}, all[kSegCounters] = {};
    for (int b = threadIdx.x; b < nblocks; b += blockDim.x)
#pragma unroll
      for (int q = 0; q < kSegCounters; ++q) {
        const int x = counts[kSegCounters * b + q];
        all[q] += x;
        if (b < (int)blockIdx.x) pre[q] += x;
      }
#pragma unroll
    for (int q = 0; q < kSegCounters; ++q) {
      int x = pre[q], y = all[q];
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        x += __shfl_xor_sync(0xffffffffu, x, o);
        y += __shfl_xor_sync(0xffffffffu, y, o);
      }
      if ((threadIdx.x & 31) == 0) {
        if (x != 0) atomicAdd(&pre_s[q], x);
        if (y != 0) atomicAdd(&all_s[q], y);
      }
    }
  }
  __syncthreads();
  const int64_t r0 = (int64_t)blockIdx.x * kScanRows + (int64_t)threadIdx.x * kRowsPerThread;
  int v[kSegCounters] = {};
  for (int i = 0; i < kRowsPerThread; ++i) {
    const int64_t r = r0 + i;
    if (r < nrows) count_row(pos[r + 1] - pos[r], v);
  }
  int at[kSegCounters];
#pragma unroll
  for (int q = 0; q < kSegCounters; ++q) at[q] = v[q];
  int tot[kSegCounters];
  block_scan<kSegCounters>(v, tot);
  // at[q]: this thread's first position of counter q (classes: within the
  // whole list, after the classes that come before it)
  int cls_start = 0;
#pragma unroll
  for (int q = 0; q < kSegCounters; ++q) {
    at[q] = pre_s[q] + v[q] - at[q] + (q < kSegClasses ? cls_start : 0);
    if (q < kSegClasses) cls_start += all_s[q];
  }
  auto put = [&](int n, int4 rec) {
    const int q = seg_class(n);
#pragma unroll
    for (int k = 0; k < kSegClasses; ++k)
      if (k == q) {
        if (at[k] < max_segs) segs[at[k]] = rec;
        ++at[k];
      }
  };
  for (int i = 0; i < kRowsPerThread; ++i) {
    const int64_t r = r0 + i;
    if (r >= nrows) break;
    const int p0 = pos[r], p1 = pos[r + 1];
    const int ns = segs_of(p1 - p0);
    if (ns == 1) {
      put(p1 - p0, make_int4((int)r, p0, p1, -1));
    } else {
      const int ho = at[kSegClasses], co = at[kSegClasses + 1];
      const bool fits = ho < max_heavy && co + ns <= max_chunks;
      if (fits) heavy[ho] = HeavyRow{(int)r, co, ns, 0};
      at[kSegClasses] += 1;
      at[kSegClasses + 1] += ns;
      // the ns - 1 full chunks are consecutive in the first class, then the
      // last chunk goes to its own class
      const int f0 = at[0];
      at[0] += ns - 1;
      for (int c = 0; c < ns - 1; ++c)
        if (f0 + c < max_segs)
          segs[f0 + c] = make_int4((int)r, p0 + c * kSegChunk, p0 + (c + 1) * kSegChunk, fits ? co + c : -1);
      const int a = p0 + (ns - 1) * kSegChunk;
      put(p1 - a, make_int4((int)r, a, p1, fits ? co + ns - 1 : -1));
    }
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    int ns = 0;
#pragma unroll
    for (int q = 0; q < kSegClasses; ++q) ns += all_s[q];
    const int nh = all_s[kSegClasses], nc = all_s[kSegClasses + 1];
    hdr->n_segs = ns;
    hdr->n_heavy = nh;
    hdr->n_chunks = nc;
    if (ns > max_segs || nh > max_heavy || nc > max_chunks) atomicOr(&hdr->error, kErrOverflow);
  }
}

// Waits until *count >= target (a monotonic shared-memory counter); false
// after `limit` clock cycles.
__device__ __forceinline__ bool count_wait_timeout(const int* count, int target, long long limit) {
  const long long t0 = clock64();
  while (tc::ld_acquire_smem(count) < target) {
    __nanosleep(64);  // leave the issue slots to the warps that are working
    if (clock64() - t0 > limit) return false;
  }
  return true;
}

#ifndef SLNR_TC_MBAR_SLEEP
#define SLNR_TC_MBAR_SLEEP 256  // back-off (ns) between polls of an mbarrier by the MMA and epilogue warps
#endif

// Waits for the phase with the given parity to complete; false after `limit`
// clock cycles.  Sleeps between polls so that the waiting MMA and epilogue
// warps leave the issue slots to the producers (their work has the slack of
// a whole tile).
__device__ __forceinline__ bool mbar_wait_timeout(uint64_t* bar, uint32_t parity, long long limit) {
  const long long t0 = clock64();
  while (!tc::mbar_try_wait(bar, parity)) {
    if (SLNR_TC_MBAR_SLEEP > 0) __nanosleep(SLNR_TC_MBAR_SLEEP);
    if (clock64() - t0 > limit) return false;
  }
  return true;
}

// Waits for the phase with the given parity to complete (1), or until
// *end <= j, i.e. there is no tile j to wait for (0); -1 after `limit` cycles.
__device__ __forceinline__ int mbar_wait_or_end(uint64_t* bar, uint32_t parity, const int* end, int j,
                                                long long limit) {
  const long long t0 = clock64();
  while (!tc::mbar_try_wait(bar, parity)) {
    if (*reinterpret_cast<const volatile int*>(end) <= j) return 0;
    if (SLNR_TC_MBAR_SLEEP > 0) __nanosleep(SLNR_TC_MBAR_SLEEP);
    if (clock64() - t0 > limit) return -1;
  }
  return 1;
}

// kSegments: gathered row segments; kSegmentsH: the same with Hadamard rows
// X[k,:] .* X2[k,:] (<SpMMH,GEMM>); kDense: rows of a materialised T.
// kSampled (<SDDMM,SpMM,GEMM>): the row of stored (i,j) is F(j,:) scaled by
// the sampled product B(i,j) <C(i,:), D(j,:)>.
enum TcMode { kSegments = 0, kDense = 1, kSegmentsH = 2, kSampled = 3 };

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

// Tensor memory columns a CTA allocates: its NBUF accumulators (L columns
// each), at least the 32 columns an allocation takes.
__host__ __device__ constexpr uint32_t tc_tmem_cols(int K, int L) {
  return tc_nbuf(K, L) * L < 32 ? 32u : (uint32_t)(tc_nbuf(K, L) * L);
}

// Epilogue staging: each of the four epilogue warps stages its 32 rows, one
// column chunk of min(L, 32) values at a time, in shared memory with a row
// pitch padded by 16 bytes (the warp's 16-byte stores of 32 different rows
// then hit every bank evenly), and reads them back transposed so that each
// global store instruction writes whole 128-byte row pieces: 4 rows of 32
// values per instruction instead of 32 scattered 16-byte pieces (one lane
// per row).  Two stages per warp where shared memory allows, else one.
__host__ __device__ constexpr int tc_chunk(int L) { return L < 32 ? L : 32; }
__host__ __device__ constexpr int tc_pitch(int L) { return tc_chunk(L) * 4 + 16; }
__host__ __device__ constexpr size_t tc_stage_bytes(int L) { return (size_t)4 * 32 * tc_pitch(L); }
__host__ __device__ constexpr size_t tc_td_bytes(int K, int L) {
  return (size_t)tc_nbuf(K, L) * kTcRows * tc_kt(K) * 4 + (size_t)L * tc_kt(K) * 4;
}
__host__ __device__ constexpr int tc_nstage(int K, int L) {
  return tc_td_bytes(K, L) + 2 * tc_stage_bytes(L) + 1024 <= (size_t)220 * 1024 ? 2 : 1;
}

// Shared memory: NBUF T tiles (kTcRows x KT) and D^T (L x KT), tf32 K-major
// 128B-swizzled, then the epilogue stages, plus 1 KB of alignment slack.
__host__ __device__ constexpr size_t tc_smem_bytes(int K, int L) {
  return tc_td_bytes(K, L) + tc_nstage(K, L) * tc_stage_bytes(L) + 1024;
}

#ifndef SLNR_TC_BATCH
#define SLNR_TC_BATCH 4  // gathered rows a lane group keeps in flight (one batch; half with Hadamard rows)
#endif
constexpr int kBatch = SLNR_TC_BATCH;
#ifndef SLNR_TC_SHORT_BATCH
#define SLNR_TC_SHORT_BATCH 8  // rows in flight in a wave of short items (they need no accumulator of their own)
#endif
constexpr int kShortBatch = SLNR_TC_SHORT_BATCH;

#ifndef SLNR_TC_STREAM_HINT
#define SLNR_TC_STREAM_HINT 1  // 1: streamed loads and stores carry an L2 evict-first hint
#endif

// Loads and stores of data each call streams through once (coordinates,
// values, segment records, output rows).  With SLNR_TC_STREAM_HINT they are
// marked evict-first in L2, so that they make room before the gathered rows,
// which are read again.
__device__ __forceinline__ uint64_t stream_policy() {
  uint64_t pol = 0;
  if (SLNR_TC_STREAM_HINT) asm("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}
__device__ __forceinline__ int ld_stream(const int32_t* p, uint64_t pol) {
  if (!SLNR_TC_STREAM_HINT) return __ldg(p);
  int v;
  asm volatile("ld.global.nc.L2::cache_hint.b32 %0, [%1], %2;" : "=r"(v) : "l"(p), "l"(pol));
  return v;
}
__device__ __forceinline__ float ld_stream(const float* p, uint64_t pol) {
  if (!SLNR_TC_STREAM_HINT) return __ldg(p);
  float v;
  asm volatile("ld.global.nc.L2::cache_hint.f32 %0, [%1], %2;" : "=f"(v) : "l"(p), "l"(pol));
  return v;
}
__device__ __forceinline__ void st_stream(float* p, float4 x, uint64_t pol) {
  if (!SLNR_TC_STREAM_HINT) {
    *reinterpret_cast<float4*>(p) = x;
    return;
  }
  asm volatile("st.global.L2::cache_hint.v4.f32 [%0], {%1, %2, %3, %4}, %5;" ::"l"(p), "f"(x.x), "f"(x.y), "f"(x.z),
               "f"(x.w), "l"(pol)
               : "memory");
}


// Producer lane layout: a T row is built by a group of GS = K / 4 lanes (at
// most a warp), lane gl of the group holding the 4 columns [4 gl, 4 gl + 4)
// as one float4; a warp holds G = 32 / GS groups.  A claim is IPC = G * R
// consecutive items of an item tile, group g taking items g R .. g R + R - 1,
// with R = min(GS, RB) (a lane of the group holds each item's record).  A
// claim's items run one after the other in each group, so the tiles of
// heavy-row chunks at the head of the list take R items' time on the claims
// of one tile; with narrow groups (many per warp) larger claims made those
// tiles the kernel's tail.  Measured on the 2^20-row R-MAT graph: R = 1 at
// K = 16 (0.55 -> 0.45 ms against R = 4), R = 2 at K = 32 (0.51 -> 0.42 ms
// against R = 8), the short-wave width 8 at K >= 64, and 4 for sampled rows,
// where every item runs on its own (8 doubled the heavy tiles' length).
template <int K, bool SEQ>
struct ProdLayout {
  static constexpr int VPL = K > 128 ? 8 : 4;  // a group is at most a warp
  static constexpr int GS = K / VPL;
  static constexpr int G = 32 / GS;
  static constexpr int RB = G >= 8 ? 1 : G == 4 ? 2 : SEQ ? kBatch : kShortBatch;
  static constexpr int R = GS < RB ? GS : RB;
  static constexpr int IPC = G * R;
  static_assert(GS >= 1 && GS <= 32 && 32 % GS == 0, "a group is a power-of-two part of a warp");
  static_assert(kTcRows % IPC == 0, "claims tile the item tile");
  static_assert(R <= GS, "each item record is held by one lane of its group");
};

// Row k of the gathered matrix, the VPL columns of this lane: X[k, col..] (or
// X[k, col..] .* X2[k, col..] with H, the product formed in fp32).
template <int K, int VPL, bool H>
__device__ __forceinline__ void gathered_row(float (&x)[VPL], const float* __restrict__ X,
                                             const float* __restrict__ X2, int c, int col) {
  ldg_vec<VPL>(x, X + (int64_t)c * K + col);
  if constexpr (H) {
    float x2[VPL];
    ldg_vec<VPL>(x2, X2 + (int64_t)c * K + col);
#pragma unroll
    for (int e = 0; e < VPL; ++e) x[e] *= x2[e];
  }
}

// Stores the VPL values of this lane's columns of T row s (buffer sTb),
// rounded to tf32, into the 128B-swizzled K-major tile.
template <int VPL>
__device__ __forceinline__ void store_t_part(uint8_t* sTb, int s, int col, const float (&acc)[VPL]) {
#pragma unroll
  for (int h = 0; h < VPL / 4; ++h)
    *reinterpret_cast<uint4*>(sTb + tc::sw128_offset(s, col + 4 * h, kTcRows)) =
        make_uint4(tc::to_tf32(acc[4 * h]), tc::to_tf32(acc[4 * h + 1]), tc::to_tf32(acc[4 * h + 2]),
                   tc::to_tf32(acc[4 * h + 3]));
}

// Segment record of item `item` ({row, p0, p1, partial slot}); items past the
// list are {-1, 0, 0, -1}: no destination, no nonzeros.
__device__ __forceinline__ int4 seg_rec(const int4* __restrict__ segs, int item, int nitems) {
  return item < nitems ? __ldg(segs + item) : make_int4(-1, 0, 0, -1);
}

// The producer gathers below run in one lane group (GS lanes, mask gmask,
// first lane gbase, this lane gl).  The group's R items are held one record
// per lane: lane gl < R holds the p0 (rp0) and p1 (rp1) of item gl and its
// destination (rdst: A row, partial slot).  Coordinates and values are loaded
// cooperatively, one nonzero per lane, and handed to the gathering lanes with
// shuffles inside the group.  Finished T rows are placed through `pl`
// (completion-order slots, see the kernel): pl.take(n) returns the first of
// n consecutive slots once their buffer is free (-1 after a timeout),
// pl.put / pl.put_dest store a row and its destination, pl.publish(sl, n)
// fences and arrives on the slot tiles' barriers.  Both return false after a
// timeout.

// A wave of W short items (items w0 .. w0 + W - 1, at most N nonzeros each,
// W N <= kBatch): lane t loads the coordinate and value of slot t (nonzero
// t % N of item t / N), all W N gathered rows are in flight at once, then
// each item's T row is summed in nonzero order and placed.
template <int K, int VPL, int GS, int W, int N, bool H, typename Place>
__device__ __forceinline__ bool short_wave(unsigned gmask, int gbase, int gl, int rp0, int rp1, int2 rdst, int w0,
                                           const int32_t* __restrict__ crd, const float* __restrict__ vals,
                                           const float* __restrict__ X, const float* __restrict__ X2, int col,
                                           Place& pl) {
  constexpr int S = W * N;                // row slots of the batch
  constexpr int SPL = (S + GS - 1) / GS;  // slots loaded per lane
  static_assert(S <= kShortBatch, "a wave is one batch");
  int mc[SPL];
  float mv[SPL];
#pragma unroll
  for (int h = 0; h < SPL; ++h) {
    const int t = gl + h * GS, w = t / N < W ? t / N : W - 1, s = t % N;
    const int p0 = __shfl_sync(gmask, rp0, gbase + w0 + w), p1 = __shfl_sync(gmask, rp1, gbase + w0 + w);
    const bool ok = t < S && p0 + s < p1;
    const uint64_t pol = stream_policy();
    mc[h] = ok ? ld_stream(crd + p0 + s, pol) : -1;
    mv[h] = ok ? ld_stream(vals + p0 + s, pol) : 0.f;
  }
  float x[S][VPL];
#pragma unroll
  for (int u = 0; u < S; ++u) {
    const int c = __shfl_sync(gmask, mc[u / GS], gbase + u % GS);
    if (c >= 0) gathered_row<K, VPL, H>(x[u], X, X2, c, col); else zero_vec(x[u]);
  }
  // each item's sum, in nonzero order, into the registers of its first row
#pragma unroll
  for (int w = 0; w < W; ++w)
#pragma unroll
    for (int s = 0; s < N; ++s) {
      const int u = w * N + s;
      const float v = __shfl_sync(gmask, mv[u / GS], gbase + u % GS);
#pragma unroll
      for (int e = 0; e < VPL; ++e) x[w * N][e] = s == 0 ? v * x[u][e] : fmaf(v, x[u][e], x[w * N][e]);
    }
  const int sl = pl.take(W);
  if (sl < 0) return false;
  return pl.template place<W>(sl, [&](int w, int slot) {
    pl.put(slot, x[w * N]);
    if (gl == w0 + w) pl.put_dest(slot, rdst);
  });
}

// The group's R items one after the other, each T row summed in nonzero
// order in batches of B gathered rows and placed when complete.  The items'
// nonzeros are walked in chunks of GS (a chunk never spans two items): lane
// t holds the coordinate and value of nonzero t of the current chunk, and the
// next chunk's (which may be the next item's first) are loaded while this one
// is gathered.  (Prefetching the next chunk's rows into L2 as well raised the
// DRAM traffic of gathered matrices larger than L2: lines arrived early and
// were evicted before use.)
// With S (sampled rows, <SDDMM,SpMM,GEMM>) the row of nonzero (i,j) is
// X(j,:) = F(j,:) scaled by y = vals <Cq(i,:), X2(j,:)>: the item's row of Cq
// stays in registers, the dot product is summed across the group by shuffles.
template <int K, int VPL, int GS, int R, bool H, bool S, typename Place>
__device__ __forceinline__ bool long_items(unsigned gmask, int gbase, int gl, int rp0, int rp1, int2 rdst,
                                           const int32_t* __restrict__ crd, const float* __restrict__ vals,
                                           const float* __restrict__ X, const float* __restrict__ X2,
                                           const float* __restrict__ Cq, int col, Place& pl) {
  constexpr bool TWO = H || S;  // two gathered rows per nonzero
  constexpr int B0 = (TWO ? kBatch / 2 : kBatch) * 4 / VPL > 0 ? (TWO ? kBatch / 2 : kBatch) * 4 / VPL : 1;  // the same registers for any row width and with two rows
  constexpr int B = B0 < GS ? B0 : GS;
  static_assert(GS % B == 0, "batches tile a chunk");
  auto p0_of = [&](int r) { return __shfl_sync(gmask, rp0, gbase + r); };
  auto p1_of = [&](int r) { return __shfl_sync(gmask, rp1, gbase + r); };
  // a chunk is item r's nonzeros [q, min(q + GS, p1(r))); r == R: none left
  auto advance = [&](int& r, int& q) {
    if (r < R && q + GS < p1_of(r)) {
      q += GS;
    } else {
      ++r;
      q = r < R ? p0_of(r) : 0;
    }
  };
  auto load_idx = [&](int r, int q, int& ic, float& iv) {
    const bool ok = r < R && q + gl < p1_of(r);
    const uint64_t pol = stream_policy();
    ic = ok ? ld_stream(crd + q + gl, pol) : -1;
    iv = ok ? ld_stream(vals + q + gl, pol) : 0.f;
  };
  int r = 0, q = p0_of(0);  // current chunk
  int rn = r, qn = q;       // next chunk
  advance(rn, qn);
  int ic, nc;
  float iv, nv;
  load_idx(r, q, ic, iv);
  load_idx(rn, qn, nc, nv);
  float acc[VPL];
  zero_vec(acc);
  float crow[S ? VPL : 1];  // S: Cq's row of the current item
  auto load_crow = [&](int rr) {
    if constexpr (S) {
      const int row = __shfl_sync(gmask, rdst.x, gbase + (rr < R ? rr : 0));
      if (rr < R && row >= 0) ldg_vec<VPL>(crow, Cq + (int64_t)row * K + col); else zero_vec(crow);
    }
  };
  load_crow(0);
#pragma unroll 1
  while (r < R) {
    const int m = min(GS, p1_of(r) - q);
#pragma unroll 1
    for (int u0 = 0; u0 < m; u0 += B) {
      float x[B][VPL];
      if constexpr (S) {
        float d[B][VPL];
#pragma unroll
        for (int k = 0; k < B; ++k) {
          const int c = __shfl_sync(gmask, ic, gbase + u0 + k);
          if (c >= 0) {
            ldg_vec<VPL>(x[k], X + (int64_t)c * K + col);
            ldg_vec<VPL>(d[k], X2 + (int64_t)c * K + col);
          } else {
            zero_vec(x[k]);
            zero_vec(d[k]);
          }
        }
#pragma unroll
        for (int k = 0; k < B; ++k) {
          float dot = 0.f;
#pragma unroll
          for (int e = 0; e < VPL; ++e) dot = fmaf(crow[e], d[k][e], dot);
#pragma unroll
          for (int o = GS / 2; o > 0; o >>= 1) dot += __shfl_xor_sync(gmask, dot, o);
          const float y = __shfl_sync(gmask, iv, gbase + u0 + k) * dot;
#pragma unroll
          for (int e = 0; e < VPL; ++e) acc[e] = fmaf(y, x[k][e], acc[e]);
        }
      } else {
#pragma unroll
        for (int k = 0; k < B; ++k) {
          const int c = __shfl_sync(gmask, ic, gbase + u0 + k);
          if (c >= 0) gathered_row<K, VPL, H>(x[k], X, X2, c, col); else zero_vec(x[k]);
        }
#pragma unroll
        for (int k = 0; k < B; ++k) {
          const float v = __shfl_sync(gmask, iv, gbase + u0 + k);
#pragma unroll
          for (int e = 0; e < VPL; ++e) acc[e] = fmaf(v, x[k][e], acc[e]);
        }
      }
    }
    if (rn != r) {  // the item's last chunk: its T row is complete
      const int sl = pl.take(1);  // one slot: always inside one slot tile
      if (sl < 0) return false;
      pl.put(sl, acc);
      if (gl == r) pl.put_dest(sl, rdst);
      pl.publish(sl, 1);
      zero_vec(acc);
      if constexpr (S) load_crow(rn);
    }
    r = rn;
    q = qn;
    ic = nc;
    iv = nv;
    advance(rn, qn);
    load_idx(rn, qn, nc, nv);
  }
  return true;
}

constexpr int kTileRing = 16;  // local tiles whose global index is kept in shared memory
constexpr int kMaxBuf = 4;     // T / accumulator buffers at most

// Shared state of the tile kernel's pipeline (one per CTA; static shared
// memory, named directly by the helpers below).
struct TcShared {
  uint64_t full_bar[kMaxBuf];  // slot tile b filled: one arrival per placed T row
  uint64_t mma_bar[kMaxBuf];   // the tile's MMAs completed (tcgen05.commit)
  uint64_t free_bar[kMaxBuf];  // the four epilogue warps have drained accumulator b
  int2 dest[kMaxBuf][kTcRows]; // per slot: (A row, partial slot); x < 0 = no destination
  uint32_t tmem_base;
  int claim;                   // next producer claim of this CTA
  int fill;                    // next T slot (completion order)
  int fail_flag;               // a wait timed out: every role winds down
  int epi_progress[4];         // per epilogue warp: tiles whose destinations it has read
  int tile_gid[kTileRing];     // global item tile of local tile j (ring)
  int tile_seq[kTileRing];     // j + 1 once tile_gid of local tile j is written
  int end_tile;                // first local tile past the last item tile
  int last_commit[kMaxBuf];    // last tile committed to each accumulator (-1: none)
  float* epi_dst[4][32];       // per epilogue warp: destination of each of its 32 rows (nullptr: none)
};
__shared__ TcShared g_tc;
extern __shared__ uint8_t smem_raw[];

// Waits until every epilogue warp has read the destinations of `tiles` slot
// tiles (each warp publishes its own count: a sum would let one warp that
// runs ahead stand in for one that lags); false after `limit` clock cycles.
__device__ __forceinline__ bool epi_wait_timeout(int tiles, long long limit) {
  const long long t0 = clock64();
  for (;;) {
    int m = tc::ld_acquire_smem(&g_tc.epi_progress[0]);
#pragma unroll
    for (int q = 1; q < 4; ++q) m = min(m, tc::ld_acquire_smem(&g_tc.epi_progress[q]));
    if (m >= tiles) return true;
    __nanosleep(64);
    if (clock64() - t0 > limit) return false;
  }
}

// The T tiles: NBUF buffers at the first 1024-byte boundary of the dynamic
// shared memory, then D^T.
__device__ __forceinline__ uint8_t* tc_tiles() {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
}

// Completion-order placement of one lane group's T rows: slots are taken
// from the CTA's fill counter after the rows are built; slot s lives in slot
// tile s / kTcRows, buffer (s / kTcRows) % NBUF.
template <int VPL, int NBUF, int TBYTES>
struct Placer {
  unsigned gmask;
  int gbase, gl, col;
  long long wait_cycles;
  // First of n consecutive slots, once the buffer of its slot tile is free
  // (all four epilogue warps have read the destinations of the tile NBUF
  // before, so its MMAs are done); -1 after a timeout.  The range may run
  // into the next slot tile: place() fills it tile by tile.
  __device__ __forceinline__ int take(int n) {
    int sl = 0;
    if (gl == 0) sl = atomicAdd(&g_tc.fill, n);
    sl = __shfl_sync(gmask, sl, gbase);
    return wait_tile(sl / kTcRows) ? sl : -1;
  }
  // Waits until slot tile t's buffer is free; false after a timeout.
  __device__ __forceinline__ bool wait_tile(int t) {
    if (t < NBUF) return true;
    const bool ok = epi_wait_timeout(t - NBUF + 1, wait_cycles);
    if (__any_sync(gmask, !ok)) {
      if (gl == 0) atomicOr(&g_tc.fail_flag, 1);
      return false;
    }
    return true;
  }
  // Stores rows 0 .. W-1 into slots sl .. sl + W - 1 (store(w, slot) puts
  // row w and its destination) and publishes them.  The rows in the first
  // slot tile are published before waiting for the next tile's buffer: with
  // one buffer that wait needs the first tile consumed, which needs them.
  template <int W, typename F>
  __device__ __forceinline__ bool place(int sl, F&& store) {
    const int n1 = min(W, kTcRows - sl % kTcRows);
#pragma unroll
    for (int w = 0; w < W; ++w)
      if (w < n1) store(w, sl + w);
    publish(sl, n1);
    if (n1 < W) {
      if (!wait_tile(sl / kTcRows + 1)) return false;
#pragma unroll
      for (int w = 0; w < W; ++w)
        if (w >= n1) store(w, sl + w);
      publish(sl + n1, W - n1);
    }
    return true;
  }
  __device__ __forceinline__ void put(int slot, const float (&acc)[VPL]) {
    store_t_part<VPL>(tc_tiles() + ((slot / kTcRows) % NBUF) * TBYTES, slot % kTcRows, col, acc);
  }
  __device__ __forceinline__ void put_dest(int slot, int2 d) { g_tc.dest[(slot / kTcRows) % NBUF][slot % kTcRows] = d; }
  // The rows (and destinations) of slots [sl, sl + n), all in one slot tile,
  // are stored: make them visible to the tensor cores and count them on the
  // tile's barrier.
  __device__ __forceinline__ void publish(int sl, int n) {
    tc::fence_proxy_async_smem();
    __syncwarp(gmask);
    if (gl == 0) tc::mbar_arrive_n(&g_tc.full_bar[(sl / kTcRows) % NBUF], (uint32_t)n);
  }
};

// Warp roles of the persistent tile kernel (kTcWarps warps):
//   producers    (all but the last five warps): take claims of IPC
//                consecutive items of this CTA's item tiles (in order) and
//                build the items' T rows with one lane group per item; each
//                finished row (or wave of short rows) takes the next T slots
//                in completion order, waits until the slots' buffer is free,
//                and is stored with its destination; one arrival per placed
//                row on the slot tile's mbarrier (kTcRows per tile);
//   MMA warp     waits full[b] (the slot tile is complete) and free[b] (the
//                buffer's previous accumulator drained), issues the tile's
//                K/8 tcgen05.mma into TMEM accumulator b, commits to mma[b];
//   4 epilogue   wait mma[b], read their destinations and publish their own
//   warps        progress (epi_progress), read their TMEM lane quadrant
//                (warp % 4), stage the rows in shared memory and write them
//                (A rows, or partial rows of heavy rows) with coalesced
//                stores of whole row pieces, arrive free[b].
// Slot tile j uses buffer j % NBUF; a row goes into it only after all four
// epilogue warps have read the destinations of slot tile j - NBUF (so its
// MMAs are done).  A CTA fills exactly as many slot tiles as it takes item
// tiles (every item, padding included, takes one slot).  Slots are taken
// after the rows are built, so a producer waits only for an earlier slot
// tile, whose slots were all taken by warps that already hold their rows and
// wait only for still earlier tiles: no cycle.  Every wait is bounded by
// wait_cycles; a timeout raises kErrTimeout and the CTA winds down (MMAs
// already issued are drained with the default limit before the tensor
// memory is freed).
constexpr int kProducerWarps = kTcWarps - 5;
constexpr int kMmaWarp = kTcWarps - 5;  // then the four epilogue warps

template <int K, int L, int MODE>
__global__ void __launch_bounds__(kTcThreads, 1)
    k_tc_gemm(WsHeader* hdr, const int4* __restrict__ segs, int max_segs,
              int64_t dense_rows, const int32_t* __restrict__ crd, const float* __restrict__ vals,
              const float* __restrict__ X, const float* __restrict__ X2, const float* __restrict__ Cq,
              const float* __restrict__ D, float* __restrict__ A, float* __restrict__ partial, long long wait_cycles) {
  static_assert(K == 16 || K == 32 || K == 64 || K == 128 || K == 256, "K must be 16, 32, 64, 128 or 256");
  static_assert(L % 16 == 0 && L >= 16 && L <= 256, "L must be a multiple of 16 in [16, 256]");
  constexpr int KT = tc_kt(K);  // tile columns (K, or 32 with zero padding)
  using PL = ProdLayout<K, MODE == kSampled>;
  constexpr int NBUF = tc_nbuf(K, L);
  constexpr uint32_t IDESC = tc::idesc_tf32(kTcRows, L);
  // TMEM columns: NBUF fp32 accumulators of L columns; an allocation is a
  // power of two of at least 32 columns
  constexpr uint32_t NCOLS = tc_tmem_cols(K, L);
  static_assert(NCOLS >= (uint32_t)(NBUF * L) && NCOLS >= 32 && (NCOLS & (NCOLS - 1)) == 0 && NCOLS <= 512,
                "tensor memory allocation");
  constexpr int TBYTES = kTcRows * KT * 4;
  constexpr int CPT = kTcRows / PL::IPC;  // claims per item tile
  static_assert(NBUF <= kMaxBuf, "buffers");
  uint8_t* sT = tc_tiles();
  uint8_t* sD = sT + NBUF * TBYTES;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (warp == kMmaWarp) {
    tc::tmem_alloc(&g_tc.tmem_base, NCOLS);
    tc::tmem_relinquish();
  }
  if (tid == 0) {
    for (int b = 0; b < NBUF; ++b) {
      tc::mbar_init(&g_tc.full_bar[b], kTcRows);  // one arrival per placed T row
      tc::mbar_init(&g_tc.mma_bar[b], 1);
      tc::mbar_init(&g_tc.free_bar[b], 4);
      g_tc.last_commit[b] = -1;
    }
    tc::fence_mbar_init();
    g_tc.claim = 0;
    g_tc.fill = 0;
    g_tc.fail_flag = 0;
    for (int q = 0; q < 4; ++q) g_tc.epi_progress[q] = 0;
  }
  // Item tiles are handed out dynamically: CTAs take them from a global
  // counter in the workspace header (zeroed before the launch), one tile
  // ahead of need, so the costly tiles do not pile up on a few SMs.  Local
  // tile j's global index is published in a small shared ring (g_tc.tile_gid,
  // with g_tc.tile_seq = j + 1 once written); the first local tile whose index
  // lies past the last item tile is g_tc.end_tile, and every role stops there.
  int nitems;  // < 2^31: segments or rows
  if (MODE != kDense) {
    const int n = hdr->n_segs;
    nitems = n < max_segs ? n : max_segs;
  } else {
    nitems = (int)dense_rows;
  }
  const int ntiles = (int)(((int64_t)nitems + kTcRows - 1) / kTcRows);
  if (tid == 0) {
    for (int r = 0; r < kTileRing; ++r) g_tc.tile_seq[r] = 0;
    const int g0 = atomicAdd(&hdr->next_tile, 1);
    g_tc.tile_gid[0] = g0;
    g_tc.tile_seq[0] = 1;
    g_tc.end_tile = g0 >= ntiles ? 0 : INT_MAX;
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
  const uint32_t tmem = g_tc.tmem_base;

  // global item tile of local tile t: >= 0 once known, -1 if t does not
  // exist (t >= g_tc.end_tile), -2 if the wait timed out
  auto tile_of = [&](int t) -> int {
    const long long t0 = clock64();
    while (tc::ld_acquire_smem(&g_tc.tile_seq[t % kTileRing]) != t + 1) {
      if (*reinterpret_cast<volatile int*>(&g_tc.end_tile) <= t) return -1;
      __nanosleep(32);
      if (clock64() - t0 > wait_cycles) return -2;
    }
    const int gid = *reinterpret_cast<volatile int*>(&g_tc.tile_gid[t % kTileRing]);
    return gid < ntiles ? gid : -1;
  };
  // the first g_tc.claim of local tile t fetches the global index of tile t + 1
  auto fetch_next_tile = [&](int t) {
    const int gnext = atomicAdd(&hdr->next_tile, 1);
    g_tc.tile_gid[(t + 1) % kTileRing] = gnext;
    if (gnext >= ntiles) atomicMin(&g_tc.end_tile, t + 1);
    tc::st_release_smem(&g_tc.tile_seq[(t + 1) % kTileRing], t + 2);
  };

  if (warp < kProducerWarps) {
    // ---------------- producers ----------------
    constexpr int VPL = PL::VPL, R = PL::R, GS = PL::GS;
    const int g = lane / GS, gl = lane % GS, col = gl * VPL, gbase = g * GS;
    const unsigned gmask = GS == 32 ? 0xffffffffu : (((1u << GS) - 1u) << gbase);
    Placer<VPL, NBUF, TBYTES> pl{gmask, gbase, gl, col, wait_cycles};
    int known_tile = -1, known_gid = -1;  // the last local tile this warp resolved
    for (;;) {
      int c = 0;
      if (lane == 0) c = atomicAdd(&g_tc.claim, 1);
      c = __shfl_sync(0xffffffffu, c, 0);
      const int j = c / CPT;
      if (j != known_tile) {
        known_gid = __shfl_sync(0xffffffffu, tile_of(j), 0);
        known_tile = known_gid >= 0 ? j : -1;
      }
      const int gid = known_gid;
      if (gid < 0) {
        if (gid == -2) atomicOr(&g_tc.fail_flag, 1);
        break;
      }
      if (c % CPT == 0) {
        if (lane == 0) fetch_next_tile(j);
        __syncwarp();
      }
      if (*reinterpret_cast<volatile int*>(&g_tc.fail_flag) != 0) break;  // another role timed out
      const int item0 = gid * kTcRows + (c % CPT) * PL::IPC + g * R;  // this group's first item
      bool ok = true;
      if constexpr (MODE == kDense) {
        // R rows of the materialised T, all loads in flight at once
        float x[R][VPL];
#pragma unroll
        for (int r = 0; r < R; ++r) {
          if (item0 + r < nitems) ldg_vec<VPL>(x[r], X + (int64_t)(item0 + r) * K + col); else zero_vec(x[r]);
        }
        const int sl = pl.take(R);
        ok = sl >= 0 && pl.template place<R>(sl, [&](int r, int slot) {
          pl.put(slot, x[r]);
          if (gl == r) pl.put_dest(slot, make_int2(item0 + r < nitems ? item0 + r : -1, -1));
        });
      } else {
        constexpr bool H = MODE == kSegmentsH;
        // lane gl < R holds the record of the group's item gl
        int rp0 = 0, rp1 = 0;
        int2 rdst = make_int2(-1, -1);
        if (gl < R) {
          const int4 rec = seg_rec(segs, item0 + gl, nitems);
          rp0 = rec.y;
          rp1 = rec.z;
          rdst = make_int2(rec.x, rec.w);
        }
        // The list is sorted by length class, longest first: no item after
        // item0 has more nonzeros than item0's class bound, so item0 picks
        // the wave shape for the group's R items.
        // rows in flight per group: fewer with two loads each (H) or 8 columns per lane
        constexpr int BW = (H ? kShortBatch / 2 : kShortBatch) * 4 / VPL > 0
                               ? (H ? kShortBatch / 2 : kShortBatch) * 4 / VPL : 1;
        constexpr int W1 = R < BW ? R : BW;
        constexpr int W2 = R < BW / 2 ? R : (BW / 2 > 1 ? BW / 2 : 1);
        constexpr int W4 = R < BW / 4 ? R : (BW / 4 > 1 ? BW / 4 : 1);
        const int n0 = __shfl_sync(gmask, rp1 - rp0, gbase);
        if (MODE == kSampled) {  // items one after the other (each keeps its C row)
          ok = long_items<K, VPL, GS, R, false, true>(gmask, gbase, gl, rp0, rp1, rdst, crd, vals, X, X2, Cq,
                                                           col, pl);
        } else if (n0 <= 1) {
#pragma unroll 1
          for (int w0 = 0; w0 < R && ok; w0 += W1)
            ok = short_wave<K, VPL, GS, W1, 1, H>(gmask, gbase, gl, rp0, rp1, rdst, w0, crd, vals, X, X2, col, pl);
        } else if (n0 <= 2) {
#pragma unroll 1
          for (int w0 = 0; w0 < R && ok; w0 += W2)
            ok = short_wave<K, VPL, GS, W2, 2, H>(gmask, gbase, gl, rp0, rp1, rdst, w0, crd, vals, X, X2, col, pl);
        } else if (n0 <= 4) {
#pragma unroll 1
          for (int w0 = 0; w0 < R && ok; w0 += W4)
            ok = short_wave<K, VPL, GS, W4, 4, H>(gmask, gbase, gl, rp0, rp1, rdst, w0, crd, vals, X, X2, col, pl);
        } else {
          ok = long_items<K, VPL, GS, R, H, false>(gmask, gbase, gl, rp0, rp1, rdst, crd, vals, X, X2, nullptr,
                                                        col, pl);
        }
      }
      if (!__all_sync(0xffffffffu, ok)) break;
    }
  } else if (warp == kMmaWarp) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      const uint32_t sT_addr = tc::smem_u32(sT), sD_addr = tc::smem_u32(sD);
      for (int j = 0;; ++j) {
        const int b = j % NBUF;
        const int st = mbar_wait_or_end(&g_tc.full_bar[b], (j / NBUF) & 1, &g_tc.end_tile, j, wait_cycles);
        if (st == 0) break;  // this CTA has no tile j
        if (st < 0 || (j >= NBUF && !mbar_wait_timeout(&g_tc.free_bar[b], ((j / NBUF) - 1) & 1, wait_cycles))) {
          atomicOr(&g_tc.fail_flag, 1);
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
        tc::mma_commit(&g_tc.mma_bar[b]);
        g_tc.last_commit[b] = j;
      }
    }
    __syncwarp();
  } else {
    // ---------------- epilogue ----------------
    const int q = warp & 3;  // TMEM lane quadrant of this warp
    constexpr int CW = tc_chunk(L), PITCH = tc_pitch(L), NSTAGE = tc_nstage(K, L);
    uint8_t* stage = sT + tc_td_bytes(K, L) + (size_t)q * NSTAGE * 32 * PITCH;
    int stage_i = 0;
    for (int j = 0;; ++j) {
      const int b = j % NBUF;
      const int st =
          __shfl_sync(0xffffffffu, mbar_wait_or_end(&g_tc.mma_bar[b], (j / NBUF) & 1, &g_tc.end_tile, j, wait_cycles), 0);
      if (st == 0) break;  // this CTA has no tile j
      if (st < 0) {
        atomicOr(&g_tc.fail_flag, 1);
        break;
      }
      tc::tc_fence_after_sync();
      const int rr = 32 * q + lane;
      const int2 dd = g_tc.dest[b][rr];
      // this warp has its destinations: once all four have, the slot tile may be refilled
      __syncwarp();
      if (lane == 0) tc::st_release_smem(&g_tc.epi_progress[q], j + 1);
      // the destinations of the warp's 32 rows, read back by the lanes that
      // store each row piece
      constexpr int LPRW = CW / 4, RPI = 32 / LPRW, NIT = 32 / RPI;
      g_tc.epi_dst[q][lane] =
          dd.x < 0 ? nullptr : (dd.y < 0 ? A + (int64_t)dd.x * L : partial + (int64_t)dd.y * L);
      __syncwarp();
      // each chunk of CW columns: TMEM -> registers (row `lane`) -> this
      // warp's stage -> 16-byte pieces of whole row pieces -> global
#pragma unroll 1
      for (int c = 0; c < L; c += CW) {
        float v[CW];
        if constexpr (CW == 32)
          tc::tmem_ld32(tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(b * L + c), v);
        else
          tc::tmem_ld16(tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(b * L + c), v);
        uint8_t* st = stage + (size_t)stage_i * 32 * PITCH;
#pragma unroll
        for (int i = 0; i < CW / 4; ++i)
          *reinterpret_cast<float4*>(st + (size_t)lane * PITCH + 16 * i) =
              make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
        __syncwarp();
#pragma unroll
        for (int i = 0; i < NIT; ++i) {
          const int r = RPI * i + lane / LPRW, part = lane % LPRW;
          const float4 x = *reinterpret_cast<const float4*>(st + (size_t)r * PITCH + 16 * part);
          float* d = g_tc.epi_dst[q][r];
          if (d != nullptr) st_stream(d + c + 4 * part, x, stream_policy());
        }
        stage_i = (stage_i + 1) % NSTAGE;  // with one stage, the next chunk's
        if (NSTAGE == 1) __syncwarp();     // stores wait for these reads
      }
      tc::tc_fence_before_sync();
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&g_tc.free_bar[b]);
    }
  }

  // ---- teardown: every role has finished its loop
  tc::tc_fence_before_sync();
  __syncthreads();
  if (g_tc.fail_flag) {
    // MMAs of abandoned tiles may still be running: wait (bounded, with the
    // default limit whatever wait_cycles was) for each accumulator's last
    // commit before the tensor memory is released
    if (warp == kMmaWarp && lane == 0)
      for (int b = 0; b < NBUF; ++b)
        if (g_tc.last_commit[b] >= 0) mbar_wait_timeout(&g_tc.mma_bar[b], (g_tc.last_commit[b] / NBUF) & 1, kWaitCycles);
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
  // no more resident CTAs per SM than tensor memory (512 columns) holds
  // accumulators for: a CTA waiting in tcgen05.alloc would only idle
  const int max_ctas = 512 / (int)tc_tmem_cols(K, L);
  const size_t floor_bytes = (size_t)sm_smem / (size_t)(max_ctas + 1) + 1;
  if (smem < floor_bytes) smem = floor_bytes;
  if ((e = cudaFuncSetAttribute(k_tc_gemm<K, L, MODE>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem)) !=
      cudaSuccess)
    return e;
  if ((e = cudaFuncSetAttribute(k_tc_gemm<K, L, MODE>, cudaFuncAttributePreferredSharedMemoryCarveout,
                                (int)cudaSharedmemCarveoutMaxShared)) != cudaSuccess)
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
                        const float* X2, const float* Cq, const float* D, float* A, float* partial, cudaStream_t s) {
  const long long wait = wait_limit_cycles();
#define SLNR_TC_CASE(KK, LL)                                                                              \
  if (K == KK && L == LL) {                                                                               \
    TcLaunch tl;                                                                                          \
    cudaError_t e = tc_setup<KK, LL, MODE>(&tl);                                                          \
    if (e != cudaSuccess) return e;                                                                       \
    int64_t grid = (items_upper + kTcRows - 1) / kTcRows;                                                 \
    if (grid > tl.grid_cap) grid = tl.grid_cap;                                                           \
    if (grid < 1) grid = 1;                                                                               \
    if ((e = cudaMemsetAsync(&hdr->next_tile, 0, sizeof(int), s)) != cudaSuccess) return e;               \
    k_tc_gemm<KK, LL, MODE><<<SLNR_COUNTED((unsigned)grid), kTcThreads, tl.smem, s>>>(hdr, segs, max_segs, dense_rows,  \
                                                                         crd, vals, X, X2, Cq, D, A,     \
                                                                         partial, wait);                 \
    return cudaGetLastError();                                                                            \
  }
  if constexpr (MODE == kSampled) {  // <SDDMM,SpMM,GEMM>: the widths of the benchmark range
    SLNR_TC_CASE(32, 32) SLNR_TC_CASE(32, 64) SLNR_TC_CASE(32, 128)
    SLNR_TC_CASE(64, 32) SLNR_TC_CASE(64, 64) SLNR_TC_CASE(64, 128)
    SLNR_TC_CASE(128, 32) SLNR_TC_CASE(128, 64) SLNR_TC_CASE(128, 128)
    return cudaErrorInvalidValue;
  }
  SLNR_TC_CASE(16, 16) SLNR_TC_CASE(16, 32) SLNR_TC_CASE(16, 64) SLNR_TC_CASE(16, 128) SLNR_TC_CASE(16, 256)
  SLNR_TC_CASE(32, 16) SLNR_TC_CASE(32, 32) SLNR_TC_CASE(32, 64) SLNR_TC_CASE(32, 128) SLNR_TC_CASE(32, 256)
  SLNR_TC_CASE(64, 16) SLNR_TC_CASE(64, 32) SLNR_TC_CASE(64, 64) SLNR_TC_CASE(64, 128) SLNR_TC_CASE(64, 256)
  SLNR_TC_CASE(128, 16) SLNR_TC_CASE(128, 32) SLNR_TC_CASE(128, 64) SLNR_TC_CASE(128, 128) SLNR_TC_CASE(128, 256)
  SLNR_TC_CASE(256, 16) SLNR_TC_CASE(256, 32) SLNR_TC_CASE(256, 64)
#undef SLNR_TC_CASE
  return cudaErrorInvalidValue;
}

}  // namespace

bool tc_supported(int K, int L) {
  return (K == 16 || K == 32 || K == 64 || K == 128 || (K == 256 && L <= 64)) &&
         (L == 16 || L == 32 || L == 64 || L == 128 || L == 256) &&
         tc_smem_bytes(K, L) <= (size_t)220 * 1024;
}

int seg_scan_blocks(int64_t nrows) { return (int)((nrows + kScanRows - 1) / kScanRows); }

cudaError_t launch_seg_count(const CsrView& B, const SegPlan& plan, cudaStream_t s) {
  if (B.nrows <= 0) return cudaSuccess;
  k_seg_count<<<SLNR_COUNTED(seg_scan_blocks(B.nrows)), kScanThreads, 0, s>>>(B.nrows, B.pos, plan.block_counts);
  return cudaGetLastError();
}

cudaError_t launch_seg_write(const CsrView& B, const SegPlan& plan, cudaStream_t s) {
  if (B.nrows <= 0) return cudaSuccess;
  const int nb = seg_scan_blocks(B.nrows);
  k_seg_write<<<SLNR_COUNTED(nb), kScanThreads, 0, s>>>(B.nrows, B.pos, plan.block_counts, nb, plan.hdr, plan.segs, plan.heavy,
                                          plan.max_segs, plan.max_heavy, plan.max_chunks);
  return cudaGetLastError();
}

cudaError_t launch_tc_spmm_gemm(int K, int L, const CsrView& B, const float* C, const float* D, float* A,
                                const SegPlan& plan, cudaStream_t s, const float* C2) {
  if (B.nrows <= 0) return cudaSuccess;
  if (C2 != nullptr)
    return tc_dispatch<kSegmentsH>(K, L, plan.max_segs, plan.hdr, plan.segs, plan.max_segs, 0, B.crd, B.vals, C, C2,
                                   nullptr, D, A, plan.partial, s);
  return tc_dispatch<kSegments>(K, L, plan.max_segs, plan.hdr, plan.segs, plan.max_segs, 0, B.crd, B.vals, C,
                                nullptr, nullptr, D, A, plan.partial, s);
}

bool tc_sampled_supported(int K, int L, int M) {
  return K == L && (L == 32 || L == 64 || L == 128) && (M == 32 || M == 64 || M == 128);
}

cudaError_t launch_tc_sddmm_spmm_gemm(const CsrView& B, const float* C, const float* D, const float* F, int L,
                                      const float* W, int M, float* A, const SegPlan& plan, cudaStream_t s) {
  if (B.nrows <= 0) return cudaSuccess;
  // T rows of width L: the gathered row is F(j,:), its scale C(i,:).D(j,:)
  return tc_dispatch<kSampled>(L, M, plan.max_segs, plan.hdr, plan.segs, plan.max_segs, 0, B.crd, B.vals, F, D, C,
                               W, A, plan.partial, s);
}

cudaError_t launch_tc_dense_gemm(int64_t M, int K, int L, const float* T, const float* D, float* A,
                                 WsHeader* hdr, cudaStream_t s) {
  if (M <= 0) return cudaSuccess;
  return tc_dispatch<kDense>(K, L, M, hdr, nullptr, 0, M, nullptr, nullptr, T, nullptr, nullptr, D, A, nullptr, s);
}

}  // namespace slnr
