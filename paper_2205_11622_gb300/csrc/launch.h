// Internal launchers of libslnr (C++ linkage, not exported).  Each returns
// the cudaError_t of its launch(es); the C entry points in api.cu map them to
// slnr_status.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "common.cuh"

namespace slnr {

// Counts the calling thread's kernel launches: every launch's grid argument is
// wrapped in SLNR_COUNTED; a call's count starts at 0 (slnr_timing_launches).
void note_launch();
#define SLNR_COUNTED(grid) (::slnr::note_launch(), (grid))

// A CSR-shaped view: rows with positions pos[nrows+1], coordinates crd and
// values vals.  CSF fibers are viewed this way too (rows = fibers,
// pos = pos3, crd = crd3).
struct CsrView {
  int nrows;
  int ncols;
  int64_t nnz;
  const int32_t* pos;
  const int32_t* crd;
  const float* vals;
};

// Workspace pieces used to split heavy rows (see common.cuh).
struct SplitPlan {
  WsHeader* hdr;
  HeavyRow* heavy;
  Chunk* chunks;
  float* partial;  // max_chunks x width
  int max_heavy;
  int max_chunks;
};

// Workspace pieces of the MTTKRP unit decomposition.
struct UnitPlan {
  WsHeader* hdr;
  SliceUnits* slice_units;  // [nslices]
  Unit* units;              // [max_units]
  float* partial;           // max_units x L
  int max_units;
  float* part_sums;         // max_units x L: sums of runs of kPartUnits unit partials of large slices
};

// Workspace pieces of the tensor-core path: row segments of at most
// kSegChunk nonzeros (tc_gemm.cu).
struct SegPlan {
  WsHeader* hdr;
  int* block_counts;  // kSegCounters ints per inspector block
  int4* segs;         // {row, p0, p1, partial slot or -1}
  HeavyRow* heavy;
  float* partial;     // max_chunks x L partial A rows
  int max_segs;
  int max_heavy;
  int max_chunks;
};

int device_sm_count();

// Sets the calling thread's slnr_last_error() text (api.cu).
void set_last_error(const char* msg);

// Default limit, in SM clock cycles, of every bounded device-side wait
// (about 2 s at 2 GHz).
constexpr long long kWaitCycles = 4000000000LL;
// The limit the calling thread's launches give their bounded waits
// (kWaitCycles unless slnr_set_wait_limit changed it; api.cu).
long long wait_limit_cycles();

// inspect.cu
cudaError_t launch_classify(const CsrView& B, const SplitPlan& plan, cudaStream_t s);
cudaError_t launch_csf_units(const slnr_csf3& B, const UnitPlan& plan, cudaStream_t s);
cudaError_t launch_validate_csr(const slnr_csr& B, WsHeader* hdr, cudaStream_t s);
cudaError_t launch_validate_csf(const slnr_csf3& B, WsHeader* hdr, cudaStream_t s);
// A's levels pos1, crd1, pos2, crd2 copied from B's in one launch
cudaError_t launch_copy_levels(const slnr_csf3& B, int32_t* A_pos1, int32_t* A_crd1, int32_t* A_pos2,
                               int32_t* A_crd2, cudaStream_t s);

// spmm.cu -- out[r,:] = sum_p vals[p] X[crd[p],:] (width W), and the heavy-row machinery
// (with X2 not NULL the gathered row is X[k,:] .* X2[k,:], the <SpMMH,GEMM> producer)
cudaError_t launch_spmm_rows(int W, const CsrView& B, const float* X, float* out, cudaStream_t s,
                             const float* X2 = nullptr);
cudaError_t launch_spmm_chunks(int W, const CsrView& B, const float* X, const SplitPlan& plan,
                               cudaStream_t s, const float* X2 = nullptr);
// heavy rows: out[row,:] = sum of the row's partials (width W); when D is not
// NULL the sum (width W = K) is multiplied by D (K x L) and out has width L.
cudaError_t launch_combine(int W, const SplitPlan& plan, const float* D, int L, float* out,
                           cudaStream_t s);

// gemm.cu -- fused SpMM x D over light rows; dense GEMM for the unfused variant
cudaError_t launch_spmm_gemm_tiles(int K, int L, const CsrView& B, const float* C, const float* D,
                                   float* A, int use_tf32, cudaStream_t s, const float* C2 = nullptr);
cudaError_t launch_dense_gemm(int64_t M, int K, int L, const float* T, const float* D, float* A,
                              int use_tf32, cudaStream_t s);

// tc_gemm.cu -- tcgen05 TF32 consumer contraction
bool tc_supported(int K, int L);
int seg_scan_blocks(int64_t nrows);
cudaError_t launch_seg_count(const CsrView& B, const SegPlan& plan, cudaStream_t s);
cudaError_t launch_seg_write(const CsrView& B, const SegPlan& plan, cudaStream_t s);
// (with C2 not NULL the gathered row is C[k,:] .* C2[k,:], <SpMMH,GEMM>)
cudaError_t launch_tc_spmm_gemm(int K, int L, const CsrView& B, const float* C, const float* D, float* A,
                                const SegPlan& plan, cudaStream_t s, const float* C2 = nullptr);
cudaError_t launch_tc_dense_gemm(int64_t M, int K, int L, const float* T, const float* D, float* A,
                                 WsHeader* hdr, cudaStream_t s);
// fused <SDDMM,SpMM,GEMM> on the tensor-core kernel: C nrows x K, D ncols x K,
// F ncols x L, W L x M, with K == L (the dot product and the temporary share the lane layout)
bool tc_sampled_supported(int K, int L, int M);
cudaError_t launch_tc_sddmm_spmm_gemm(const CsrView& B, const float* C, const float* D, const float* F, int L,
                                      const float* W, int M, float* A, const SegPlan& plan, cudaStream_t s);

// sddmm.cu
// fused <SDDMM,SpMM>: the heavy rows' chunks (partials) and the light rows in
// one launch (plan.hdr->next_row must be 0: warps take work from it)
cudaError_t launch_sddmm_spmm_rows(const CsrView& B, const float* C, const float* D, int L,
                                   const float* E, int K, float* A, const SplitPlan& plan, cudaStream_t s);
cudaError_t launch_sddmm_spmm_chunks(const CsrView& B, const float* C, const float* D, int L,
                                     const float* E, int K, const SplitPlan& plan, cudaStream_t s);
// fused <SDDMM,SpMM,GEMM> over light rows: C nrows x K, D ncols x K, F ncols x L, W L x M
cudaError_t launch_sddmm_spmm_gemm_tiles(const CsrView& B, const float* C, const float* D, int K,
                                         const float* F, int L, const float* W, int M, float* A, cudaStream_t s);
cudaError_t launch_sddmm_rows(const CsrView& B, const float* C, const float* D, int L, float* Y,
                              cudaStream_t s);
cudaError_t launch_sddmm_chunks(const CsrView& B, const float* C, const float* D, int L, float* Y,
                                const SplitPlan& plan, cudaStream_t s);

// mttkrp.cu
cudaError_t launch_mttkrp_units(int L, const slnr_csf3& B, const float* C, const float* D,
                                const UnitPlan& plan, cudaStream_t s);
cudaError_t launch_mttkrp_stage2_units(int L, const slnr_csf3& B, const float* T, const float* C,
                                       const UnitPlan& plan, cudaStream_t s);
// A(i,:) = sum of slice i's unit partials (width L); with E (L x M) not NULL,
// that sum times E (A has width M).
cudaError_t launch_mttkrp_combine(int L, const slnr_csf3& B, const UnitPlan& plan, const float* E, int M,
                                  float* A, cudaStream_t s);

// wide.cu -- any inner width that is a multiple of 4 up to kWideMax, chosen at
// run time (the kernels above take powers of two in [4, 256])
constexpr int kWideMax = 1024;
bool wide_dim(int d);
// out = B . X (width W; with X2, the gathered row is X .* X2): light rows to
// out, heavy rows' chunks to plan.partial (then launch_w_combine)
cudaError_t launch_w_spmm(int W, const CsrView& B, const float* X, const float* X2, float* out,
                          const SplitPlan& plan, cudaStream_t s);
// heavy rows: out[row,:] = sum of the row's partials (width W), times D (W x L) when D is not NULL
cudaError_t launch_w_combine(int W, const SplitPlan& plan, const float* D, int L, float* out, cudaStream_t s);
// fused B . C . D over light rows (T tile on chip); with C2, the gathered row is C .* C2
cudaError_t launch_w_spmm_gemm_tiles(int K, int L, const CsrView& B, const float* C, const float* C2,
                                     const float* D, float* A, cudaStream_t s);
cudaError_t launch_w_dense_gemm(int64_t M, int K, int L, const float* T, const float* D, float* A, cudaStream_t s);
// fused <SDDMM,SpMM> (C nrows x Kd, D ncols x Kd, E ncols x Ko): light rows to A,
// heavy rows' chunks to plan.partial; with Y not NULL, only the sampled products Y[p]
cudaError_t launch_w_sddmm_spmm(const CsrView& B, const float* C, const float* D, int Kd, const float* E, int Ko,
                                float* A, float* Y, const SplitPlan& plan, cudaStream_t s);
cudaError_t launch_w_sddmm_spmm_gemm_tiles(const CsrView& B, const float* C, const float* D, int K, const float* F,
                                           int L, const float* W, int M, float* A, cudaStream_t s);
// MTTKRP unit partials: fused (T == NULL) or from the per-fiber T (unfused)
cudaError_t launch_w_mttkrp_units(int L, const slnr_csf3& B, const float* C, const float* D, const float* T,
                                  const UnitPlan& plan, cudaStream_t s);
cudaError_t launch_w_mttkrp_combine(int L, const slnr_csf3& B, const UnitPlan& plan, const float* E, int M, float* A,
                                    cudaStream_t s);

// peaks.cu -- peaks measured by the library's own kernels (TFLOP/s, GB/s)
cudaError_t peak_ffma(cudaStream_t s, double* tflops);
cudaError_t peak_tf32(cudaStream_t s, double* tflops);
// rows x width fp32 table (width in {4, 8, ..., 128}, 16-byte aligned); GB/s of row gathers
cudaError_t peak_gather(const float* table, int64_t rows, int width, cudaStream_t s, double* gbs);

}  // namespace slnr

// Runs `body` with a compile-time constant WCONST equal to the runtime width
// w (a power of two in [4, 256]); any other w returns cudaErrorInvalidValue.
#define SLNR_WIDTH_SWITCH(w, WCONST, ...)                \
  switch (w) {                                           \
    case 4: { constexpr int WCONST = 4; __VA_ARGS__; } break;     \
    case 8: { constexpr int WCONST = 8; __VA_ARGS__; } break;     \
    case 16: { constexpr int WCONST = 16; __VA_ARGS__; } break;   \
    case 32: { constexpr int WCONST = 32; __VA_ARGS__; } break;   \
    case 64: { constexpr int WCONST = 64; __VA_ARGS__; } break;   \
    case 128: { constexpr int WCONST = 128; __VA_ARGS__; } break; \
    case 256: { constexpr int WCONST = 256; __VA_ARGS__; } break; \
    default: return cudaErrorInvalidValue;               \
  }
