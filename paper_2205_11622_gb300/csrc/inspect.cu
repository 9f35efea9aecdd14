// Inspector kernels (work decomposition for power-law inputs) and the
// optional device-side validation of index arrays.
//
// The paper parallelises the shared outer sparse loop with OpenMP (Sec. 2.3,
// Sec. 6) and names load imbalance from irregular structure as a core
// difficulty (Sec. 1).  On the GPU the outer loop is split by nonzero count:
// light rows are processed whole, heavy rows (more than kLightMax nonzeros)
// are cut into chunks of kChunk nonzeros whose partial results are combined
// in a fixed order, and MTTKRP slices are cut into windows of kUnitNnz
// nonzeros.
#include "launch.h"

namespace slnr {

int device_sm_count() {
  static int cached[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 148;
  if (cached[dev] == 0) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 148;
    cached[dev] = n;
  }
  return cached[dev];
}

namespace {

__global__ void k_classify(int nrows, const int32_t* __restrict__ pos, WsHeader* hdr,
                           HeavyRow* __restrict__ heavy, Chunk* __restrict__ chunks, int max_heavy,
                           int max_chunks) {
  for (int r = blockIdx.x * blockDim.x + threadIdx.x; r < nrows; r += gridDim.x * blockDim.x) {
    const int p0 = pos[r], p1 = pos[r + 1];
    const int n = p1 - p0;
    if (n <= kLightMax) continue;
    const int nch = (n + kChunk - 1) / kChunk;
    const int h = atomicAdd(&hdr->n_heavy, 1);
    const int base = atomicAdd(&hdr->n_chunks, nch);
    if (h >= max_heavy || base + nch > max_chunks) {
      atomicOr(&hdr->error, kErrOverflow);
      continue;
    }
    heavy[h] = HeavyRow{r, base, nch, 0};
    for (int c = 0; c < nch; ++c) {
      const int a = p0 + c * kChunk;
      chunks[base + c] = Chunk{r, a, min(p1, a + kChunk), base + c};
    }
  }
}

// First f in [lo, hi) with pos[f] >= key (hi if none).
__device__ __forceinline__ int lower_bound_pos(const int32_t* __restrict__ pos, int lo, int hi, int key) {
  while (lo < hi) {
    const int mid = lo + ((hi - lo) >> 1);
    if (__ldg(pos + mid) < key) lo = mid + 1; else hi = mid;
  }
  return lo;
}

// One warp per slice: the slice is cut into units, the fibers that start in
// one window of kUnitNnz nonzeros, and the lanes write the unit records.
__global__ void k_csf_units(int nslices, const int32_t* __restrict__ pos2,
                            const int32_t* __restrict__ pos3, WsHeader* hdr,
                            SliceUnits* __restrict__ su, Unit* __restrict__ units, int max_units) {
  const int lane = threadIdx.x & 31;
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t sw = warp; sw < nslices; sw += nwarps) {
    const int s = (int)sw;
    const int n = pos3[pos2[s + 1]] - pos3[pos2[s]];
    const int nu = n > 0 ? (n + kUnitNnz - 1) / kUnitNnz : 1;
    int base = 0;
    if (lane == 0) base = atomicAdd(&hdr->n_units, nu);
    base = __shfl_sync(0xffffffffu, base, 0);
    if (base + nu > max_units) {
      if (lane == 0) {
        atomicOr(&hdr->error, kErrOverflow);
        su[s] = SliceUnits{0, 0};
      }
      continue;
    }
    if (lane == 0) su[s] = SliceUnits{base, nu};
    for (int u = lane; u < nu; u += 32) units[base + u] = Unit{s, u, 0, 0, 0, 0, 0, 0};
  }
}

// One thread per unit: its nonzero window [p0, p1), the fiber holding p0,
// and the fibers of its slice whose first nonzero lies in the window
// [flo, fhi) (binary searches over pos3).
__global__ void k_unit_ranges(const WsHeader* __restrict__ hdr, int max_units, const int32_t* __restrict__ pos2,
                              const int32_t* __restrict__ pos3, const SliceUnits* __restrict__ su,
                              Unit* __restrict__ units) {
  const int n = min(hdr->n_units, max_units);
  for (int64_t w = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; w < n; w += (int64_t)gridDim.x * blockDim.x) {
    Unit un = units[w];
    const int f0 = pos2[un.slice], f1 = pos2[un.slice + 1];
    const int start = pos3[f0], count = su[un.slice].count;
    const int lo_key = start + un.u * kUnitNnz;
    un.flo = un.u == 0 ? f0 : lower_bound_pos(pos3, f0, f1, lo_key);
    un.fhi = un.u == count - 1 ? f1 : lower_bound_pos(pos3, f0, f1, lo_key + kUnitNnz);
    const int end = pos3[f1];
    un.p0 = min(lo_key, end);
    un.p1 = un.u == count - 1 ? end : min(lo_key + kUnitNnz, end);
    // the fiber holding p0: flo if it starts exactly there, else the one before
    un.ffirst = (un.flo < f1 && pos3[un.flo] == un.p0) || un.flo == f0 ? un.flo : un.flo - 1;
    units[w] = un;
  }
}

// A's compressed levels as copies of B's (<SpTTM,SpTTM>: the (i,j) pattern is
// unchanged) in one launch: pos1 (2), pos2 (nslices + 1) and crd1 (nslices)
// in a grid-stride pass over their concatenation, then crd2 (nfibers, the
// bulk) in 16-byte pieces where both arrays are 16-byte aligned.
__global__ void k_copy_levels(const int32_t* __restrict__ pos1, const int32_t* __restrict__ pos2,
                              const int32_t* __restrict__ crd1, const int32_t* __restrict__ crd2, int32_t* a_pos1,
                              int32_t* a_pos2, int32_t* a_crd1, int32_t* a_crd2, int nslices, int nfibers,
                              bool vec) {
  const int64_t tid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x, stride = (int64_t)gridDim.x * blockDim.x;
  const int64_t n0 = 2, n1 = n0 + nslices + 1, n2 = n1 + nslices;
  for (int64_t i = tid; i < n2; i += stride) {
    if (i < n0) a_pos1[i] = pos1[i];
    else if (i < n1) a_pos2[i - n0] = pos2[i - n0];
    else a_crd1[i - n1] = crd1[i - n1];
  }
  const int64_t n4 = vec ? nfibers / 4 : 0;
  for (int64_t i = tid; i < n4; i += stride)
    reinterpret_cast<int4*>(a_crd2)[i] = __ldg(reinterpret_cast<const int4*>(crd2) + i);
  for (int64_t i = 4 * n4 + tid; i < nfibers; i += stride) a_crd2[i] = crd2[i];
}

// One thread per parent: checks its position range and the order and range of
// its children's coordinates.  Ranges are clamped so a malformed array never
// leads to an out-of-bounds read.
__device__ void check_level(int parent, int nparents, const int32_t* __restrict__ pos, int64_t nchild,
                            const int32_t* __restrict__ crd, int64_t dim, int* err) {
  const int64_t a = pos[parent], b = pos[parent + 1];
  if (parent == 0 && a != 0) atomicOr(err, kErrPos);
  if (parent == nparents - 1 && b != nchild) atomicOr(err, kErrPos);
  if (a < 0 || b < a || b > nchild) {
    atomicOr(err, kErrPos);
    return;
  }
  int64_t prev = -1;
  for (int64_t p = a; p < b; ++p) {
    const int64_t c = crd[p];
    if (c < 0 || c >= dim) atomicOr(err, kErrCrdRange);
    if (c <= prev) atomicOr(err, kErrCrdOrder);
    prev = c;
  }
}

__global__ void k_validate_csr(slnr_csr B, WsHeader* hdr) {
  for (int r = blockIdx.x * blockDim.x + threadIdx.x; r < B.nrows; r += gridDim.x * blockDim.x)
    check_level(r, B.nrows, B.pos, B.nnz, B.crd, B.ncols, &hdr->error);
  if (B.nrows == 0 && blockIdx.x == 0 && threadIdx.x == 0 && (B.pos[0] != 0 || B.nnz != 0))
    atomicOr(&hdr->error, kErrPos);
}

__global__ void k_validate_csf(slnr_csf3 B, WsHeader* hdr) {
  const int tid = blockIdx.x * blockDim.x + threadIdx.x, nth = gridDim.x * blockDim.x;
  if (tid == 0) {
    if (B.pos1[0] != 0 || B.pos1[1] != B.nslices) atomicOr(&hdr->error, kErrPos);
    if (B.nslices == 0 && (B.nfibers != 0 || B.nnz != 0)) atomicOr(&hdr->error, kErrPos);
  }
  for (int q = tid; q < B.nslices; q += nth) {
    const int64_t i = B.crd1[q];
    if (i < 0 || i >= B.dim[0]) atomicOr(&hdr->error, kErrCrdRange);
    if (q > 0 && B.crd1[q - 1] >= i) atomicOr(&hdr->error, kErrCrdOrder);
    check_level(q, B.nslices, B.pos2, B.nfibers, B.crd2, B.dim[1], &hdr->error);
  }
  for (int f = tid; f < B.nfibers; f += nth)
    check_level(f, B.nfibers, B.pos3, B.nnz, B.crd3, B.dim[2], &hdr->error);
}

inline int grid_for(int64_t n, int block) {
  const int64_t cap = (int64_t)device_sm_count() * 16;
  int64_t g = (n + block - 1) / block;
  if (g > cap) g = cap;
  return (int)(g < 1 ? 1 : g);
}

}  // namespace

cudaError_t launch_classify(const CsrView& B, const SplitPlan& plan, cudaStream_t s) {
  if (B.nrows <= 0) return cudaSuccess;
  k_classify<<<SLNR_COUNTED(grid_for(B.nrows, 256)), 256, 0, s>>>(B.nrows, B.pos, plan.hdr, plan.heavy, plan.chunks,
                                                    plan.max_heavy, plan.max_chunks);
  return cudaGetLastError();
}

cudaError_t launch_csf_units(const slnr_csf3& B, const UnitPlan& plan, cudaStream_t s) {
  if (B.nslices <= 0) return cudaSuccess;
  k_csf_units<<<SLNR_COUNTED(grid_for((int64_t)B.nslices * 32, 256)), 256, 0, s>>>(B.nslices, B.pos2, B.pos3, plan.hdr,
                                                                     plan.slice_units, plan.units, plan.max_units);
  k_unit_ranges<<<SLNR_COUNTED(grid_for(plan.max_units, 256)), 256, 0, s>>>(plan.hdr, plan.max_units, B.pos2, B.pos3,
                                                               plan.slice_units, plan.units);
  return cudaGetLastError();
}

cudaError_t launch_copy_levels(const slnr_csf3& B, int32_t* A_pos1, int32_t* A_crd1, int32_t* A_pos2,
                               int32_t* A_crd2, cudaStream_t s) {
  const bool vec = (reinterpret_cast<uintptr_t>(B.crd2) & 15u) == 0 && (reinterpret_cast<uintptr_t>(A_crd2) & 15u) == 0;
  const int64_t n = 2 * (int64_t)B.nslices + 3 + (vec ? B.nfibers / 4 : B.nfibers);
  const int64_t cap = (int64_t)device_sm_count() * 8;
  int64_t grid = (n + 255) / 256;
  if (grid > cap) grid = cap;
  k_copy_levels<<<SLNR_COUNTED((unsigned)grid), 256, 0, s>>>(B.pos1, B.pos2, B.crd1, B.crd2, A_pos1, A_pos2, A_crd1, A_crd2,
                                               B.nslices, B.nfibers, vec);
  return cudaGetLastError();
}

cudaError_t launch_validate_csr(const slnr_csr& B, WsHeader* hdr, cudaStream_t s) {
  k_validate_csr<<<SLNR_COUNTED(grid_for(B.nrows > 0 ? B.nrows : 1, 256)), 256, 0, s>>>(B, hdr);
  return cudaGetLastError();
}

cudaError_t launch_validate_csf(const slnr_csf3& B, WsHeader* hdr, cudaStream_t s) {
  const int64_t n = B.nfibers > B.nslices ? B.nfibers : B.nslices;
  k_validate_csf<<<SLNR_COUNTED(grid_for(n > 0 ? n : 1, 256)), 256, 0, s>>>(B, hdr);
  return cudaGetLastError();
}

}  // namespace slnr
