// slnr_spmm_gemm_original: <SpMM,GEMM> evaluated as one perfect loop nest,
// the schedule the expression gets without SparseLNR's transformation (the
// "TACO Original" of Sec. 6; Fig. 2c shows the same kind of nest for
// <SDDMM,SpMM>): for every row i, stored B(i,j), k and l, in that order,
//   A(i,l) += B(i,j) C(j,k) D(k,l)
// with no temporary, so every (j,k) product is scaled into all L columns and
// the work is O(nnz K L), against O(nnz K + rows K L) for the fused schedule.
// It is the comparator of the inner-dimension case study (Sec. 6.3, Fig. 8b),
// not a variant of any expression of the fused path.
#include <cstdio>
#include <cstring>

#include "launch.h"

namespace {

// Lanes per row: L lanes below 32 columns (32 / L rows per warp), else 32
// lanes with CPL columns each (1, 2 or 4; a row wider than 32 CPL columns is
// split into column blocks taken by different warps).
// Each (row, column block) is a work item, grid-stride over warps; lanes
// past the warp's rows idle.  Loops i, j, k, l as in the nest; each output
// element is one fp32 chain over the row's nonzeros, then k.
template <int CPL>
__global__ void __launch_bounds__(256) k_spmm_gemm_original(int nrows, const int32_t* __restrict__ pos,
                                                            const int32_t* __restrict__ crd,
                                                            const float* __restrict__ vals,
                                                            const float* __restrict__ C, int K,
                                                            const float* __restrict__ D, int L,
                                                            float* __restrict__ A) {
  const int lane = threadIdx.x & 31;
  const int lpr = L < 32 ? L : 32, rpw = 32 / lpr, slot = lane / lpr, cl = lane % lpr;
  const int bw = lpr * CPL, nblk = (L + bw - 1) / bw;  // columns of a block, blocks per row
  const int64_t ngroups = ((int64_t)nrows + rpw - 1) / rpw;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t w = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; w < ngroups * nblk; w += nwarps) {
    const int64_t i = (w / nblk) * rpw + slot;
    const int c0 = (int)(w % nblk) * bw;
    if (slot >= rpw || i >= nrows) continue;  // no shuffles below: lanes may leave
    float acc[CPL];
#pragma unroll
    for (int u = 0; u < CPL; ++u) acc[u] = 0.f;
    for (int p = pos[i]; p < pos[i + 1]; ++p) {
      const int64_t j = crd[p];
      const float b = vals[p];
      for (int k = 0; k < K; ++k) {
        const float s = b * __ldg(C + j * K + k);
        const float* d = D + (int64_t)k * L;
#pragma unroll
        for (int u = 0; u < CPL; ++u) {
          const int l = c0 + cl + lpr * u;
          if (l < L) acc[u] = fmaf(s, __ldg(d + l), acc[u]);
        }
      }
    }
#pragma unroll
    for (int u = 0; u < CPL; ++u) {
      const int l = c0 + cl + lpr * u;
      if (l < L) A[i * L + l] = acc[u];
    }
  }
}

slnr_status fail(slnr_status st, const char* msg) {
  slnr::set_last_error(msg);
  return st;
}

}  // namespace

extern "C" slnr_status slnr_spmm_gemm_original(const slnr_csr* B, const float* C, int32_t K, const float* D,
                                                int32_t L, float* A, void* stream) {
  // B, K and L are checked as slnr_spmm_gemm checks them
  slnr_opts o;
  std::memset(&o, 0, sizeof(o));
  o.variant = SLNR_UNFUSED;
  size_t need = 0;
  const slnr_status st = slnr_spmm_gemm_workspace(B, K, L, &o, &need);
  if (st != SLNR_OK) return st;
  if (!C || !D || !A) return fail(SLNR_ERR_NULL, "slnr_spmm_gemm_original: C, D or A is NULL");
  if (B->nrows == 0) return SLNR_OK;
  const int cpl = L <= 32 ? 1 : L <= 64 ? 2 : 4;
  const int lpr = L < 32 ? L : 32, rpw = 32 / lpr;
  const int64_t warps = ((int64_t)B->nrows + rpw - 1) / rpw * ((L + lpr * cpl - 1) / (lpr * cpl));
  int64_t grid = (warps + 7) / 8;
  const int64_t cap = (int64_t)slnr::device_sm_count() * 32;
  if (grid > cap) grid = cap;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (cpl == 1)
    k_spmm_gemm_original<1><<<SLNR_COUNTED((unsigned)grid), 256, 0, s>>>(B->nrows, B->pos, B->crd, B->vals, C, K,
                                                                        D, L, A);
  else if (cpl == 2)
    k_spmm_gemm_original<2><<<SLNR_COUNTED((unsigned)grid), 256, 0, s>>>(B->nrows, B->pos, B->crd, B->vals, C, K,
                                                                        D, L, A);
  else
    k_spmm_gemm_original<4><<<SLNR_COUNTED((unsigned)grid), 256, 0, s>>>(B->nrows, B->pos, B->crd, B->vals, C, K,
                                                                        D, L, A);
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) {
    char msg[256];
    snprintf(msg, sizeof(msg), "slnr_spmm_gemm_original: launch failed: %s", cudaGetErrorString(e));
    return fail(SLNR_ERR_CUDA, msg);
  }
  return SLNR_OK;
}
