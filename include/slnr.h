/*
 * slnr.h -- C ABI of libslnr: fused composite sparse tensor expressions on
 * one NVIDIA GB300 (sm_103a).
 *
 * The library evaluates the four benchmark expressions of "SparseLNR:
 * Accelerating Sparse Tensor Computations Using Loop Nest Restructuring"
 * (Dias, Sundararajah, Saumya, Kulkarni; ICS'22, arXiv 2205.11622), Sec. 6.2,
 * and three further expressions of the same section, with the schedule that the paper's "loop fusion after distribution"
 * (Sec. 4.2, Algorithm 1) derives: the outer sparse loop (CSR row, or CSF
 * slice / fiber) is shared by the producer and the consumer, the producer
 * fills a small temporary (a scalar or a vector) and the consumer uses it at
 * once, so the intermediate tensor is never written to memory.  Each entry
 * point also has an UNFUSED variant that materialises the intermediate in the
 * caller's workspace and runs producer and consumer as separate kernels (the
 * paper's "TACO Separate" baseline, Sec. 6); slnr_spmm_gemm_original runs
 * <SpMM,GEMM> as the perfect loop nest (its "TACO Original").
 *
 * Conventions shared by every entry point
 *  - Every array argument (sparse structure, dense operands, outputs,
 *    workspace) is a DEVICE pointer owned by the caller.  The library never
 *    allocates or frees device memory.
 *  - Dense operands and outputs are fp32, row-major, densely packed (leading
 *    dimension = number of columns), and 16-byte aligned.
 *  - Index arrays are int32; coordinates are sorted ascending and unique
 *    within each parent (row, slice or fiber); every nnz count is < 2^31.
 *  - Inner dimensions (K, L, M, J) may be any multiple of 4 in [4, 1024];
 *    other values return SLNR_ERR_UNSUPPORTED.  Powers of two in [4, 256]
 *    run on kernels specialised for their width (TF32 tensor cores for the
 *    dense contractions of the fused <SpMM,GEMM>, <SpTTM,SpTTM> and
 *    <SpMMH,GEMM> with K in {16, 32, 64, 128}, or K = 256 with L <= 64);
 *    other widths on kernels that take the width at run time, with the same
 *    schedules.
 *  - Work is enqueued on opts->stream (a cudaStream_t; NULL = the legacy
 *    default stream) and runs asynchronously: the call returns once the
 *    kernels are enqueued.  With opts->validate != 0 the call first checks the
 *    index arrays on the device, waits for that check on the stream, and
 *    returns SLNR_ERR_INDEX (enqueuing nothing else) if they are malformed.
 *    With validate == 0 the indices are trusted; malformed indices are then
 *    undefined behaviour.  In validate mode the call also waits for its
 *    kernels at the end and returns SLNR_ERR_TIMEOUT if a bounded device-side
 *    wait gave up (see slnr_set_wait_limit).
 *  - opts->workspace must hold at least the number of bytes that the
 *    matching slnr_*_workspace query reports for the same arguments, and be
 *    256-byte aligned.  Its contents need no initialisation; calls that share
 *    one workspace must not overlap in time.
 *  - Every element of every output is written (rows, slices or fibers with
 *    no stored nonzero get zeros).  Outputs must not alias any input.
 *  - Host-side argument checks are synchronous and happen before any launch.
 *    On an error nothing is enqueued (except SLNR_ERR_CUDA, raised by a
 *    failed launch) and slnr_last_error() describes it.
 */
#ifndef SLNR_H
#define SLNR_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum slnr_status {
  SLNR_OK = 0,
  SLNR_ERR_NULL = 1,        /* a required pointer is NULL */
  SLNR_ERR_SHAPE = 2,       /* inconsistent or negative sizes */
  SLNR_ERR_INDEX = 3,       /* validate mode found malformed index arrays */
  SLNR_ERR_WORKSPACE = 4,   /* workspace missing, too small or misaligned */
  SLNR_ERR_UNSUPPORTED = 5, /* valid input outside what the kernels support */
  SLNR_ERR_CUDA = 6,        /* a CUDA runtime call or launch failed */
  SLNR_ERR_TIMEOUT = 7      /* a bounded device-side wait gave up */
} slnr_status;

typedef enum slnr_variant {
  SLNR_FUSED = 0,  /* shared outer sparse loop, temporary kept on chip */
  SLNR_UNFUSED = 1 /* producer and consumer as separate kernels, intermediate in workspace */
} slnr_variant;

/* Sparse matrix in CSR (the paper's format for the 2-D expressions, Sec. 6.2):
 * row i holds coordinates crd[pos[i] .. pos[i+1]) with values vals[same]. */
typedef struct slnr_csr {
  int32_t nrows, ncols;
  int64_t nnz;        /* == pos[nrows] */
  const int32_t *pos; /* [nrows + 1] */
  const int32_t *crd; /* [nnz] */
  const float *vals;  /* [nnz] */
} slnr_csr;

/* Sparse 3-tensor B(i,j,k) in CSF, levels i -> j -> k, all compressed
 * (the paper's format for the 3-D expressions, Sec. 6.2). */
typedef struct slnr_csf3 {
  int32_t dim[3];      /* d0 x d1 x d2 */
  int64_t nnz;         /* == pos3[nfibers] */
  int32_t nslices;     /* stored i coordinates (== pos1[1]) */
  int32_t nfibers;     /* stored (i,j) pairs (== pos2[nslices]) */
  const int32_t *pos1; /* [2] = {0, nslices} */
  const int32_t *crd1; /* [nslices]   i */
  const int32_t *pos2; /* [nslices+1] */
  const int32_t *crd2; /* [nfibers]   j */
  const int32_t *pos3; /* [nfibers+1] */
  const int32_t *crd3; /* [nnz]       k */
  const float *vals;   /* [nnz] */
} slnr_csf3;

typedef struct slnr_opts {
  int32_t variant;        /* slnr_variant */
  int32_t allow_tf32;     /* nonzero: dense contractions may run on TF32 tensor cores */
  int32_t validate;       /* nonzero: check index arrays on the device first (synchronises) */
  int32_t reserved;       /* must be 0 */
  void *stream;           /* cudaStream_t */
  void *workspace;        /* device scratch, >= the queried size, 256-byte aligned */
  size_t workspace_bytes; /* size of workspace */
} slnr_opts;

/* ---- workspace queries -------------------------------------------------
 * Bytes of workspace the matching call needs for these sizes and options
 * (variant changes it).  Depends only on the sizes and counts in the
 * structure descriptor, never on device data.  Pointers in B may be NULL.
 * Returns SLNR_OK and writes *bytes, or an argument error. */
slnr_status slnr_spmm_gemm_workspace(const slnr_csr *B, int32_t K, int32_t L, const slnr_opts *opts,
                                     size_t *bytes);
slnr_status slnr_sddmm_spmm_workspace(const slnr_csr *B, int32_t L, int32_t K, const slnr_opts *opts,
                                      size_t *bytes);
slnr_status slnr_mttkrp_workspace(const slnr_csf3 *B, int32_t L, const slnr_opts *opts, size_t *bytes);
slnr_status slnr_spttm_ttm_workspace(const slnr_csf3 *B, int32_t L, int32_t M, const slnr_opts *opts,
                                     size_t *bytes);
slnr_status slnr_sddmm_spmm_gemm_workspace(const slnr_csr *B, int32_t K, int32_t L, int32_t M,
                                           const slnr_opts *opts, size_t *bytes);
slnr_status slnr_mttkrp_gemm_workspace(const slnr_csf3 *B, int32_t L, int32_t M, const slnr_opts *opts,
                                       size_t *bytes);
slnr_status slnr_spmmh_gemm_workspace(const slnr_csr *B, int32_t J, int32_t L, const slnr_opts *opts,
                                      size_t *bytes);

/* ---- <SpMM,GEMM>  (Sec. 6.2; case study Sec. 6.3) ----------------------
 * A(i,l) = sum_{j,k} B(i,j) * C(j,k) * D(k,l)
 *   B: nrows x ncols CSR.  C: ncols x K.  D: K x L.  A: nrows x L (output).
 * Fused: per row i, the temporary T(k) = sum_j B(i,j) C(j,k) is built on chip
 * and multiplied by D at once (the vector temporary over k of Sec. 6.3).
 * Unfused: T = B.C is written to the workspace (nrows x K), then A = T.D.
 * With allow_tf32 the T.D contraction may use TF32 tensor cores. */
slnr_status slnr_spmm_gemm(const slnr_csr *B, const float *C, int32_t K, const float *D, int32_t L,
                           float *A, const slnr_opts *opts);

/* ---- <SDDMM,SpMM>  (Sec. 3.1 motivating example, Fig. 2; Sec. 6.2) -----
 * A(i,k) = sum_j B(i,j) * (sum_l C(i,l) * D(j,l)) * E(j,k)
 *   B: nrows x ncols CSR.  C: nrows x L.  D: ncols x L.  E: ncols x K.
 *   A: nrows x K (output).  (The paper writes the inner indices as k for the
 *   dot product and l for the output; only the names differ.)
 * Fused: per stored (i,j) the scalar y = B(i,j) C(i,:).D(j,:) is formed and
 * used at once (Fig. 2d).  Unfused: the sampled product Y (nnz values) is
 * written to the workspace, then A = Y.E (Fig. 2a then 2b). */
slnr_status slnr_sddmm_spmm(const slnr_csr *B, const float *C, const float *D, int32_t L,
                            const float *E, int32_t K, float *A, const slnr_opts *opts);

/* ---- MTTKRP  (Sec. 6.2, the MTTKRP part of <MTTKRP,GEMM>) --------------
 * A(i,l) = sum_{j,k} B(i,j,k) * C(j,l) * D(k,l)
 *   B: d0 x d1 x d2 CSF.  C: d1 x L.  D: d2 x L.  A: d0 x L (output).
 * Fused: per fiber (i,j) the temporary T(l) = sum_k B(i,j,k) D(k,l) is built
 * on chip and A(i,:) += T .* C(j,:) follows at once.  Unfused: T for every
 * fiber (nfibers x L) is written to the workspace first. */
slnr_status slnr_mttkrp(const slnr_csf3 *B, const float *C, const float *D, int32_t L, float *A,
                        const slnr_opts *opts);

/* ---- <SpTTM,SpTTM>  (Sec. 6.2, Fig. 6) ---------------------------------
 * A(i,j,m) = sum_{k,l} B(i,j,k) * C(k,l) * D(l,m),  A sparse in (i,j), dense in m.
 *   B: d0 x d1 x d2 CSF.  C: d2 x L.  D: L x M.
 * Outputs: A's compressed levels, which equal B's first two levels
 *   (A_pos1[2], A_crd1[nslices], A_pos2[nslices+1], A_crd2[nfibers]), and
 *   A_vals (nfibers x M, row f belongs to B's fiber f).
 * Fused: per fiber the temporary T(l) = sum_k B(i,j,k) C(k,l) is built on chip
 * and multiplied by D at once.  Unfused ("separate1" of Sec. 6.2): T for every
 * fiber is written to the workspace, then A_vals = T.D.  With allow_tf32 the
 * T.D contraction may use TF32 tensor cores. */
slnr_status slnr_spttm_ttm(const slnr_csf3 *B, const float *C, int32_t L, const float *D, int32_t M,
                           int32_t *A_pos1, int32_t *A_crd1, int32_t *A_pos2, int32_t *A_crd2,
                           float *A_vals, const slnr_opts *opts);

/* ---- <SDDMM,SpMM,GEMM>  (Sec. 6.2; recursive fusion, Sec. 4.2) ---------
 * A(i,m) = sum_{j,k,l} B(i,j) * C(i,k) * D(j,k) * F(j,l) * W(l,m)
 *   B: nrows x ncols CSR.  C: nrows x K.  D: ncols x K.  F: ncols x L.
 *   W: L x M.  A: nrows x M (output).
 * Fused: Algorithm 1 applied twice.  Per row i, per stored (i,j) the scalar
 * y = B(i,j) C(i,:).D(j,:) is formed and T(i,:) += y F(j,:) at once; the row's
 * vector temporary T(i,:) (length L) stays on chip and A(i,:) = T(i,:).W
 * follows: on TF32 tensor cores with allow_tf32 when K == L in {32, 64, 128}
 * and M in {32, 64, 128}, else fp32 FFMA.  Unfused: the sampled product Y (nnz values) and
 * T = Y.F (nrows x L) are written to the workspace, then A = T.W (TF32 tensor
 * cores with allow_tf32, where the widths allow). */
slnr_status slnr_sddmm_spmm_gemm(const slnr_csr *B, const float *C, const float *D, int32_t K, const float *F,
                                 int32_t L, const float *W, int32_t M, float *A, const slnr_opts *opts);

/* ---- <MTTKRP,GEMM>  (Sec. 6.2) ------------------------------------------
 * A(i,m) = sum_{j,k,l} B(i,j,k) * C(j,l) * D(k,l) * E(l,m)
 *   B: d0 x d1 x d2 CSF.  C: d1 x L.  D: d2 x L.  E: L x M.  A: d0 x M (output).
 *   (The paper writes the rank index as j: A_im = sum B_ikl C_lj D_kj E_jm.)
 * Fused: as slnr_mttkrp, and each slice's MTTKRP row u(i,:) (length L) is
 * formed on chip and multiplied by E at once (fp32 FFMA); rows without a
 * slice are zero.  Unfused: the MTTKRP result (d0 x L) is written to the
 * workspace (itself by the unfused MTTKRP schedule), then A = result.E. */
slnr_status slnr_mttkrp_gemm(const slnr_csf3 *B, const float *C, const float *D, int32_t L, const float *E,
                             int32_t M, float *A, const slnr_opts *opts);

/* ---- <SpMMH,GEMM>  (Sec. 6.2) -------------------------------------------
 * A(i,l) = sum_{k,j} B(i,k) * C(k,j) * D(k,j) * E(j,l)
 *   B: nrows x ncols CSR.  C, D: ncols x J.  E: J x L.  A: nrows x L (output).
 * Fused: per row i the temporary T(j) = sum_k B(i,k) C(k,j) D(k,j) (a sparse
 * row times the Hadamard product of the gathered rows) is built on chip and
 * multiplied by E at once, as in <SpMM,GEMM>.  Unfused: T (nrows x J) is
 * written to the workspace, then A = T.E.  With allow_tf32 the T.E
 * contraction may use TF32 tensor cores. */
slnr_status slnr_spmmh_gemm(const slnr_csr *B, const float *C, const float *D, int32_t J, const float *E,
                            int32_t L, float *A, const slnr_opts *opts);

/* ---- <SDDMM,SpMM> without a caller workspace ----------------------------
 * The paper has no counterpart to this entry point; it serves callers that
 * cannot allocate device memory (a real-time or signal-safe path that must
 * not enter an allocator, which can block or take locks, or a host runtime
 * that owns all device memory and hands none to the libraries it hosts).  It runs the fused variant of
 * slnr_sddmm_spmm with the same arguments and results, but its scratch is a
 * 16 MiB array inside the library's device code: every GPU that loads the
 * library holds those 16 MiB until the process exits, and the call allocates
 * nothing.  Sizes whose scratch would exceed 16 MiB (about 7 million nonzeros
 * at K = 64) return SLNR_ERR_UNSUPPORTED.  The first call on each device
 * looks up the array's device address (cudaGetSymbolAddress) with that device
 * current and keeps it.  A device reset (cudaDeviceReset) leaves the kept address stale:
 * do not call this entry point on a device after resetting it.  All calls
 * share the one array: the call clears what must start at zero itself, and
 * calls whose work overlaps on the GPU (other streams, other host threads)
 * race on it.  Runs on `stream` (a cudaStream_t, NULL = legacy default), with
 * validate off and fp32 arithmetic. */
slnr_status slnr_sddmm_spmm_noalloc(const slnr_csr *B, const float *C, const float *D, int32_t L,
                                    const float *E, int32_t K, float *A, void *stream);

/* ---- comparator: <SpMM,GEMM> as the perfect loop nest ---------------------
 * A(i,l) = sum_{j,k} B(i,j) C(j,k) D(k,l) evaluated with the loops i, j, k, l
 * nested in that order and no temporary: the schedule without SparseLNR's
 * transformation ("TACO Original" in Sec. 6), O(nnz K L) work.  It is the
 * comparator of the inner-dimension case study (Sec. 6.3, Fig. 8b), not a
 * variant of the fused path.  Arguments and layout as slnr_spmm_gemm (B, K
 * and L are checked the same way; C, D, A device pointers, A written
 * whole); fp32 arithmetic, one chain per output element over the row's
 * nonzeros and then k.  Needs no workspace; runs on `stream` (NULL = legacy
 * default) asynchronously. */
slnr_status slnr_spmm_gemm_original(const slnr_csr *B, const float *C, int32_t K, const float *D, int32_t L,
                                    float *A, void *stream);

/* ---- per-launch timing (instrumentation) --------------------------------
 * With timing enabled, each call on the calling thread records a CUDA event on
 * opts->stream before each of its phases (a named step of one or two kernel
 * launches) and one after the last, so phase i's device duration is the time
 * between events i and i+1.  A call overwrites the previous call's record.
 * Reading a duration waits for the call's last event.  Costs one event record
 * per phase; off by default. */
slnr_status slnr_timing_enable(int32_t on);
/* Phases recorded by the calling thread's last call (0 if timing is off). */
int32_t slnr_timing_count(void);
/* Name of phase i of the last call and its device time in milliseconds. */
slnr_status slnr_timing_get(int32_t i, const char **name, float *ms);
/* Kernel launches of the calling thread's last call (or of the call in
 * progress), counted whether timing is on or not.  Memsets and copies the
 * call enqueues are not kernels of this library and are not counted. */
int32_t slnr_timing_launches(void);

/* ---- bounded device-side waits ------------------------------------------
 * Every spin of the tensor-core kernels (on an mbarrier, a shared counter or
 * the tile-index ring) gives up after a limit of SM clock cycles, sets the
 * timeout bit of the workspace flag word and winds the CTA down (MMAs
 * already issued are drained, with the default limit, before the tensor
 * memory is freed).  A call with opts->validate != 0 waits for its launches
 * and returns SLNR_ERR_TIMEOUT when that bit is set.  This sets the limit
 * that the calling thread's later calls give those waits: cycles = 0
 * restores the default (4e9 cycles, about 2 s at 2 GHz).  Meant for testing
 * the timeout path; a limit shorter than the work makes correct calls fail.
 * Returns SLNR_ERR_SHAPE for cycles < 0. */
slnr_status slnr_set_wait_limit(int64_t cycles);

/* ---- compute peaks --------------------------------------------------------
 * The GPU's FP32 FFMA rate (CUDA cores) and TF32 rate (tcgen05 tensor cores,
 * kind::tf32, M = 128, N = 256), each measured by a kernel of this library
 * (a second, timed launch after a first one), in TFLOP/s.  They are the
 * compute denominators of the roofline the benchmark reports; neither is
 * part of any expression.  Runs on `stream` (NULL = legacy default) and
 * waits for it; allocates nothing.  slnr_peak_tf32 returns SLNR_ERR_TIMEOUT
 * if its bounded wait for the MMAs gave up. */
slnr_status slnr_peak_ffma(void *stream, double *tflops);
slnr_status slnr_peak_tf32(void *stream, double *tflops);

/* The rate of whole-row gathers, the loads the fused producers issue for
 * each nonzero (Sec. 6.3: the fused <SpMM,GEMM> reads one row of C per
 * nonzero), in GB/s: lane groups of width/4 lanes read rows of the caller's
 * device table (rows x width fp32, row-major, 16-byte aligned, contents
 * arbitrary; not written) at pseudo-random row ids, 8 rows in flight per
 * group, about 4 GB per launch; a second, timed launch follows a first one.
 * A table that fits in L2 gives the L2 gather rate, a larger one the HBM
 * gather rate.  width is a power of two in [4, 128] and rows in
 * [1, 2^31) (SLNR_ERR_SHAPE otherwise); a misaligned table returns
 * SLNR_ERR_UNSUPPORTED.  Runs on `stream` and waits for it; allocates
 * nothing. */
slnr_status slnr_peak_gather(const float *table, int64_t rows, int width, void *stream, double *gbs);

/* ---- diagnostics ------------------------------------------------------- */
const char *slnr_status_string(slnr_status status);
/* Detail of the last error raised on the calling thread ("" if none). */
const char *slnr_last_error(void);
/* Library version string. */
const char *slnr_version(void);

#ifdef __cplusplus
}
#endif

#endif /* SLNR_H */
