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

__device__ __forceinline__ bool mbar_wait_timeout(uint64_t* bar, uint32_t parity) {
  const long long t0 = clock64();
  while (!tc::mbar_try_wait(bar, parity))
    if (clock64() - t0 > kWaitCycles) return false;
  return true;
}

enum TcMode { kSegments = 0, kDense = 1 };

// Number of T / accumulator buffers: up to four, as many as fit beside D^T
// in shared memory (200 KB budget) and in tensor memory (512 columns).
__host__ __device__ constexpr int tc_nbuf(int K, int L) {
  return ((size_t)4 * kTcRows * K * 4 + (size_t)L * K * 4 + 1024 <= (size_t)200 * 1024 && 4 * L <= 512) ? 4 : 2;
}

// Shared memory: NBUF T tiles (kTcRows x K) and D^T (L x K), tf32 K-major
// 128B-swizzled, plus 1 KB of alignment slack.
__host__ __device__ constexpr size_t tc_smem_bytes(int K, int L) {
  return (size_t)tc_nbuf(K, L) * kTcRows * K * 4 + (size_t)L * K * 4 + 1024;
}

#ifndef SLNR_TC_ROWS_IN_FLIGHT
#define SLNR_TC_ROWS_IN_FLIGHT 8  // gathered rows of X in flight per producer warp (K <= 64)
#endif
#ifndef SLNR_TC_ROWS_IN_FLIGHT_K128
#define SLNR_TC_ROWS_IN_FLIGHT_K128 4  // the same for K = 128 (register budget)
#endif

// Producer layout: a whole warp builds one T row at a time (no divergence
// inside a warp); lane l holds the F = K/32 consecutive values
// [F*l, F*l + F), loaded as one float / float2 / float4, so each gathered
// row is one coalesced warp load.  U rows are in flight per warp (build-time
// defaults below).  A claim is
// kQuad consecutive items (segments), whose nonzeros form one contiguous
// range.
template <int K>
struct ProdLayout {
  static constexpr int F = K / 32;
  static constexpr int U = K >= 128 ? SLNR_TC_ROWS_IN_FLIGHT_K128 : SLNR_TC_ROWS_IN_FLIGHT;
};
constexpr int kQuad = 4;

template <int F>
struct Frag {
  float v[F];
};

template <int F>
__device__ __forceinline__ Frag<F> ldg_frag(const float* __restrict__ p) {
  Frag<F> r;
  if constexpr (F == 4) {
    const float4 a = __ldg(reinterpret_cast<const float4*>(p));
    r.v[0] = a.x; r.v[1] = a.y; r.v[2] = a.z; r.v[3] = a.w;
  } else if constexpr (F == 2) {
    const float2 a = __ldg(reinterpret_cast<const float2*>(p));
    r.v[0] = a.x; r.v[1] = a.y;
  } else {
    r.v[0] = __ldg(p);
  }
  return r;
}

template <int F>
__device__ __forceinline__ Frag<F> zero_frag() {
  Frag<F> r;
#pragma unroll
  for (int e = 0; e < F; ++e) r.v[e] = 0.f;
  return r;
}

// T row s of buffer sTb, lane's values [F*lane, F*lane+F), rounded to tf32.
template <int K>
__device__ __forceinline__ void store_t_row(uint8_t* sTb, int s, int lane, const Frag<K / 32>& acc) {
  constexpr int F = K / 32;
  uint8_t* dst = sTb + tc::sw128_offset(s, F * lane, kTcRows);
  if constexpr (F == 4) {
    *reinterpret_cast<uint4*>(dst) =
        make_uint4(tc::to_tf32(acc.v[0]), tc::to_tf32(acc.v[1]), tc::to_tf32(acc.v[2]), tc::to_tf32(acc.v[3]));
  } else if constexpr (F == 2) {
    *reinterpret_cast<uint2*>(dst) = make_uint2(tc::to_tf32(acc.v[0]), tc::to_tf32(acc.v[1]));
  } else {
    *reinterpret_cast<uint32_t*>(dst) = tc::to_tf32(acc.v[0]);
  }
}

// Accumulates the kQuad rows of one claim: row q sums vals[p] X[crd[p],:] over
// its range, which ends at the value lane q holds in my_end; the ranges are
// consecutive from p, so one pipeline of U row gathers runs over all of them,
// and emit(q, acc) hands each row on as soon as its range is done (returns
// false to abandon the claim).  Coordinates and values of the next batch are
// fetched while the current rows are in flight, one nonzero per lane, and
// passed on by shuffles.
template <int K, int U, typename Emit>
__device__ __forceinline__ bool build_quad(int my_end, int p, int lane, const int32_t* __restrict__ crd,
                                           const float* __restrict__ vals, const float* __restrict__ X,
                                           Emit&& emit) {
  constexpr int F = K / 32;
  static_assert(U <= 32 && kQuad <= 32, "one lane per prefetched nonzero and per row");
  const int p_end = __shfl_sync(0xffffffffu, my_end, kQuad - 1);
  Frag<F> acc = zero_frag<F>();
  int q = 0;
  int cur_end = __shfl_sync(0xffffffffu, my_end, 0);
  int my_c = 0;
  float my_v = 0.f;
  if (lane < U && p + lane < p_end) {
    my_c = __ldg(crd + p + lane);
    my_v = __ldg(vals + p + lane);
  }
  while (p < p_end) {
    float v[U];
    Frag<F> x[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int cu = __shfl_sync(0xffffffffu, my_c, u);
      v[u] = __shfl_sync(0xffffffffu, my_v, u);
      x[u] = (p + u < p_end) ? ldg_frag<F>(X + (int64_t)cu * K + F * lane) : zero_frag<F>();
    }
    const int pn = p + U;
    my_c = 0;
    my_v = 0.f;
    if (lane < U && pn + lane < p_end) {
      my_c = __ldg(crd + pn + lane);
      my_v = __ldg(vals + pn + lane);
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      if (p + u < p_end) {
        while (p + u >= cur_end) {  // rows whose range is complete (empty rows included)
          if (!emit(q, acc)) return false;
          acc = zero_frag<F>();
          ++q;
          cur_end = __shfl_sync(0xffffffffu, my_end, q);
        }
#pragma unroll
        for (int e = 0; e < F; ++e) acc.v[e] = fmaf(v[u], x[u].v[e], acc.v[e]);
      }
    }
    p = pn;
  }
  for (; q < kQuad; ++q) {
    if (!emit(q, acc)) return false;
    acc = zero_frag<F>();
  }
  return true;
}

// Warp roles of the persistent tile kernel (32 warps):
//   warps 0..26  producers: claim kQuad of this CTA's items at a time, build
//                their T rows on chip, and put each finished row into the next
//                free slot of the open T buffer, recording its destination;
//                MMA tiles are thus filled in completion order, so a long
//                segment delays only its own row, never a whole tile;
//   warp 27      MMA issuer: waits full[b] (128 rows placed) and free[b]
//                (buffer's previous accumulator drained), issues the tile's
//                K/8 tcgen05.mma into TMEM accumulator b, commits to mma[b];
//   warps 28..31 epilogue: wait mma[b], read TMEM lane quadrant (warp % 4),
//                write A rows or partial rows, arrive free[b].
// Slot tile n uses buffer n % NBUF; a producer fills it only after the MMAs
// of tile n - NBUF completed.  Producers may run ahead further than an
// mbarrier's phase parity can tell apart, so they wait on mma_tiles_done, a
// monotonic count of completed tiles that the epilogue publishes (release)
// once all four epilogue warps have read the tile's row destinations.
// Every wait is bounded; a timeout raises kErrTimeout and the CTA winds down.
constexpr int kProducerWarps = 27;
constexpr int kMmaWarp = 27;  // warps 28..31: epilogue

template <int K, int L, int MODE>
__global__ void __launch_bounds__(kTcThreads, 1)
    k_tc_gemm(WsHeader* hdr, const int4* __restrict__ segs, int max_segs,
              int64_t dense_rows, const int32_t* __restrict__ crd, const float* __restrict__ vals,
              const float* __restrict__ X, const float* __restrict__ D, float* __restrict__ A,
              float* __restrict__ partial) {
  static_assert(K % 32 == 0 && K >= 32 && K <= 128, "K must be 32, 64 or 128");
  static_assert(L % 32 == 0 && L >= 32 && L <= 256, "L must be a multiple of 32 in [32, 256]");
  static_assert(kTcThreads == 1024, "32 warps: 27 producers, 1 MMA, 4 epilogue");
  using PL = ProdLayout<K>;
  constexpr int F = PL::F;
  constexpr int NBUF = tc_nbuf(K, L);
  constexpr uint32_t IDESC = tc::idesc_tf32(kTcRows, L);
  constexpr uint32_t NCOLS = NBUF * L;  // TMEM columns: NBUF fp32 accumulators
  constexpr int TBYTES = kTcRows * K * 4;
  extern __shared__ uint8_t smem_raw[];
  __shared__ uint64_t full_bar[NBUF], mma_bar[NBUF], free_bar[NBUF];
  __shared__ int2 dest[NBUF][kTcRows];  // per slot: (A row, partial slot); x < 0 = padding
  __shared__ uint32_t tmem_base;
  __shared__ int claim, fill, fail_flag, mma_tiles_done;
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
      tc::mbar_init(&full_bar[b], kTcRows);
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

  int64_t nitems;
  if (MODE == kSegments) {
    const int n = hdr->n_segs;
    nitems = n < max_segs ? n : max_segs;
  } else {
    nitems = dense_rows;
  }
  const int64_t ntiles = (nitems + kTcRows - 1) / kTcRows;
  // this CTA's items: rows of item tiles blockIdx.x + j * gridDim.x, j < nlocal
  const int nlocal = (int)(ntiles > blockIdx.x ? (ntiles - blockIdx.x + gridDim.x - 1) / gridDim.x : 0);
  int total_rows = nlocal * kTcRows;
  if (nlocal > 0 && (int64_t)blockIdx.x + (int64_t)(nlocal - 1) * gridDim.x == ntiles - 1)
    total_rows -= (int)(ntiles * kTcRows - nitems);  // the global last item tile is partial
  const int pad = nlocal * kTcRows - total_rows;      // padding slots of the last slot tile

  if (warp < kProducerWarps) {
    // ---------------- producers ----------------
    constexpr int QPT = kTcRows / kQuad;  // claims per item tile
    // claim c covers local item tile c / QPT, rows (c % QPT) * kQuad + 0..kQuad-1;
    // lane q < kQuad loads the record of row q (x < 0: past the last item)
    auto load_claim = [&](int c, int4& rec) {
      rec = make_int4(-1, 0, 0, -1);
      const int64_t item =
          ((int64_t)blockIdx.x + (int64_t)(c / QPT) * gridDim.x) * kTcRows + (c % QPT) * kQuad + lane;
      if (c / QPT < nlocal && lane < kQuad && item < nitems)
        rec = (MODE == kSegments) ? __ldg(segs + item) : make_int4((int)item, 0, 0, -1);
    };
    // hands a finished T row of claimed item q to the next free slot
    int4 rec = make_int4(-1, 0, 0, -1);
    auto emit = [&](int q, const Frag<F>& acc) -> bool {
      const int rx = __shfl_sync(0xffffffffu, rec.x, q), rw = __shfl_sync(0xffffffffu, rec.w, q);
      if (rx < 0) return true;  // past the last item: no row
      int slot = 0;
      if (lane == 0) slot = atomicAdd(&fill, 1);
      slot = __shfl_sync(0xffffffffu, slot, 0);
      const int n = slot / kTcRows, s = slot % kTcRows, b = n % NBUF;
      if (n >= NBUF) {  // buffer b is free once the MMAs of slot tile n - NBUF completed
        const bool ok = count_wait_timeout(&mma_tiles_done, n - NBUF + 1);
        if (!__all_sync(0xffffffffu, ok)) return false;
      }
      store_t_row<K>(sT + b * TBYTES, s, lane, acc);
      if (lane == 0) dest[b][s] = make_int2(rx, rw);
      tc::fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) {
        if (slot == total_rows - 1 && pad > 0) {  // the last row: pad the final slot tile
          for (int i = s + 1; i < kTcRows; ++i) dest[b][i] = make_int2(-1, -1);
          tc::mbar_arrive_n(&full_bar[b], 1 + pad);
        } else {
          tc::mbar_arrive(&full_bar[b]);
        }
      }
      return true;
    };
    int x = 0;
    if (lane == 0) x = atomicAdd(&claim, 1);
    int cl = __shfl_sync(0xffffffffu, x, 0);
    load_claim(cl, rec);
    while (cl / QPT < nlocal) {
      x = 0;
      if (lane == 0) x = atomicAdd(&claim, 1);
      const int cl_next = __shfl_sync(0xffffffffu, x, 0);
      int4 rec_next;
      load_claim(cl_next, rec_next);  // loads while this claim is built
      bool ok = true;
      if (MODE == kSegments) {
        // items past the last one get an empty range at the end of the last valid item
        const unsigned valid = __ballot_sync(0xffffffffu, lane < kQuad && rec.x >= 0) & ((1u << kQuad) - 1u);
        const int nvalid = __popc(valid);
        const int start0 = __shfl_sync(0xffffffffu, rec.y, 0);
        const int last_end = __shfl_sync(0xffffffffu, rec.z, nvalid > 0 ? nvalid - 1 : 0);
        const int my_end = rec.x >= 0 ? rec.z : (nvalid > 0 ? last_end : start0);
        ok = build_quad<K, PL::U>(my_end, nvalid > 0 ? start0 : 0, lane, crd, vals, X, emit);
      } else {
#pragma unroll
        for (int q = 0; q < kQuad && ok; ++q) {
          const int rx = __shfl_sync(0xffffffffu, rec.x, q);
          const Frag<F> acc = rx >= 0 ? ldg_frag<F>(X + (int64_t)rx * K + F * lane) : zero_frag<F>();
          ok = emit(q, acc);
        }
      }
      if (!ok) {
        atomicOr(&fail_flag, 1);
        break;
      }
      cl = cl_next;
      rec = rec_next;
    }
  } else if (warp == kMmaWarp) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      const uint32_t sT_addr = tc::smem_u32(sT), sD_addr = tc::smem_u32(sD);
      for (int j = 0; j < nlocal; ++j) {
        const int b = j % NBUF;
        if (!mbar_wait_timeout(&full_bar[b], (j / NBUF) & 1) ||
            (j >= NBUF && !mbar_wait_timeout(&free_bar[b], ((j / NBUF) - 1) & 1))) {
          atomicOr(&fail_flag, 1);
          break;
        }
        tc::tc_fence_after_sync();
        const uint32_t a_base = sT_addr + b * TBYTES;
#pragma unroll
        for (int kb = 0; kb < K / 32; ++kb)
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
    for (int j = 0; j < nlocal; ++j) {
      const int b = j % NBUF;
      const bool ok = mbar_wait_timeout(&mma_bar[b], (j / NBUF) & 1);
      if (!__all_sync(0xffffffffu, ok)) {
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
  const int max_ctas = 512 / (tc_nbuf(K, L) * L);
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
  SLNR_TC_CASE(128, 32) SLNR_TC_CASE(128, 64) SLNR_TC_CASE(128, 128)
#undef SLNR_TC_CASE
  return cudaErrorInvalidValue;
}

}  // namespace

bool tc_supported(int K, int L) {
  return (K == 32 || K == 64 || K == 128) && (L == 32 || L == 64 || L == 128 || L == 256) &&
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
