/*
 * ORACLE -- test infrastructure, not part of the library.
 *
 * Plain, slow, single-threaded CPU evaluation of the four composite sparse
 * expressions of the SparseLNR paper (Dias et al., ICS'22), in fp64.  Only the
 * tests, the smoke check and the benchmark's CPU-baseline leg use it; the CUDA
 * library never includes, links or calls anything here, and nothing here
 * comes from the CUDA side.
 *
 * Every expression has a plain mathematical definition, and the paper's
 * fused schedule reaches that same value up to rounding order (Sec. 3.1.3:
 * "computes the same result"; Fig. 2 caption).  So each function below is the
 * definition written out, evaluated in the loop order that the paper's
 * "loop fusion after distribution" transformation (Sec. 4.2, Algorithm 1)
 * produces for that expression: the shared outer sparse loops, then the
 * producer loop filling a small temporary, then the consumer loop that uses
 * it.  Inputs are fp32 as stored; every product and sum is formed in double,
 * as in the paper's listings (Fig. 2, which accumulate in double).
 *
 * Each function also returns the magnitude companion A_abs: the same loops
 * applied to the absolute values of every input.  |A - A_hat| <= c * u * A_abs
 * is the standard forward error bound of any summation order, so tests
 * compare GPU results against the oracle relative to A_abs.
 *
 * Sparse formats (Sec. 6.2, "Sparse Formats"): CSR for matrices, CSF for the
 * 3-tensors; coordinates are sorted and unique within each parent.  Dense
 * operands are row-major.
 *
 * Return value of every function: 0 on success, -1 on a malformed input
 * (index out of range, non-monotone position array) or allocation failure.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

static int csr_row_ok(int32_t nrows, const int32_t *pos, int32_t i) {
  return i >= 0 && i < nrows && pos[i] <= pos[i + 1];
}

/*
 * <SpMM,GEMM> (Sec. 6.2): A(i,l) = sum_{j,k} B(i,j) * C(j,k) * D(k,l).
 *
 * Algorithm 1 removes the last operand D: the producer is T'(i,k) =
 * sum_j B(i,j) C(j,k) (loop order i, j, k) and the consumer is A(i,l) =
 * sum_k T'(i,k) D(k,l) (loop order i, k, l).  Their common loop prefix is {i};
 * below it the common index is k, so the temporary is a vector over k, live
 * for one row i (Sec. 6.3 describes exactly this "temporary vector of the
 * length of the size of dimension k").
 *
 * B: nrows x ncols CSR (pos[nrows+1], crd, vals).  C: ncols x K.  D: K x L.
 * Rows evaluated: rows[0..nsel) (or 0..nsel-1 when rows is NULL); output row s
 * of A / A_abs (nsel x L) belongs to the s-th evaluated row.
 */
int oracle_spmm_gemm(int32_t nrows, int32_t ncols, const int32_t *pos, const int32_t *crd,
                     const float *vals, const float *C, int32_t K, const float *D, int32_t L,
                     int64_t nsel, const int32_t *rows, double *A, double *A_abs) {
  double *t = (double *)malloc(sizeof(double) * (size_t)(K > 0 ? K : 1));
  double *ta = (double *)malloc(sizeof(double) * (size_t)(K > 0 ? K : 1));
  if (!t || !ta) {
    free(t);
    free(ta);
    return -1;
  }
  int rc = 0;
  for (int64_t s = 0; s < nsel && rc == 0; ++s) {
    const int32_t i = rows ? rows[s] : (int32_t)s;
    if (!csr_row_ok(nrows, pos, i)) {
      rc = -1;
      break;
    }
    /* producer: t(k) = sum_j B(i,j) C(j,k) */
    for (int32_t k = 0; k < K; ++k) {
      t[k] = 0.0;
      ta[k] = 0.0;
    }
    for (int32_t p = pos[i]; p < pos[i + 1]; ++p) {
      const int32_t j = crd[p];
      if (j < 0 || j >= ncols) {
        rc = -1;
        break;
      }
      const double b = (double)vals[p];
      for (int32_t k = 0; k < K; ++k) {
        const double c = (double)C[(int64_t)j * K + k];
        t[k] += b * c;
        ta[k] += fabs(b) * fabs(c);
      }
    }
    /* consumer: A(i,l) = sum_k t(k) D(k,l) */
    for (int32_t l = 0; l < L; ++l) {
      double acc = 0.0, acc_abs = 0.0;
      for (int32_t k = 0; k < K; ++k) {
        const double d = (double)D[(int64_t)k * L + l];
        acc += t[k] * d;
        acc_abs += ta[k] * fabs(d);
      }
      A[s * L + l] = acc;
      A_abs[s * L + l] = acc_abs;
    }
  }
  free(t);
  free(ta);
  return rc;
}

/*
 * <SDDMM,SpMM> (Sec. 3.1 and Sec. 6.2), written with the operand names of the
 * C interface: A(i,k) = sum_j B(i,j) * (sum_l C(i,l) * D(j,l)) * E(j,k).
 * (The paper names the two inner indices the other way round:
 * A_il = sum B_ij C_ik D_jk E_jl; the listings of Fig. 2 index C by row i and
 * D by column j, which is what is used here.)
 *
 * Algorithm 1 removes E: producer Y(i,j) = B(i,j) sum_l C(i,l) D(j,l) (loops
 * i, j, l), consumer A(i,k) = sum_j Y(i,j) E(j,k) (loops i, j, k).  The common
 * prefix is {i, j} and no index below it is shared, so the temporary is a
 * scalar per stored (i,j) (Sec. 4.2, "we can define the temporary as a
 * scalar"; Fig. 2d).
 *
 * B: nrows x ncols CSR.  C: nrows x L.  D: ncols x L.  E: ncols x K.
 * Output rows as for oracle_spmm_gemm; A / A_abs are nsel x K.
 */
int oracle_sddmm_spmm(int32_t nrows, int32_t ncols, const int32_t *pos, const int32_t *crd,
                      const float *vals, const float *C, const float *D, int32_t L, const float *E,
                      int32_t K, int64_t nsel, const int32_t *rows, double *A, double *A_abs) {
  for (int64_t s = 0; s < nsel; ++s) {
    const int32_t i = rows ? rows[s] : (int32_t)s;
    if (!csr_row_ok(nrows, pos, i)) return -1;
    double *a = A + s * K, *aa = A_abs + s * K;
    for (int32_t k = 0; k < K; ++k) {
      a[k] = 0.0;
      aa[k] = 0.0;
    }
    for (int32_t p = pos[i]; p < pos[i + 1]; ++p) {
      const int32_t j = crd[p];
      if (j < 0 || j >= ncols) return -1;
      const double b = (double)vals[p];
      /* producer: the scalar y = sum_l B(i,j) C(i,l) D(j,l) */
      double y = 0.0, ya = 0.0;
      for (int32_t l = 0; l < L; ++l) {
        const double c = (double)C[(int64_t)i * L + l];
        const double d = (double)D[(int64_t)j * L + l];
        y += b * c * d;
        ya += fabs(b) * fabs(c) * fabs(d);
      }
      /* consumer: A(i,k) += y E(j,k) */
      for (int32_t k = 0; k < K; ++k) {
        const double e = (double)E[(int64_t)j * K + k];
        a[k] += y * e;
        aa[k] += ya * fabs(e);
      }
    }
  }
  return 0;
}

/*
 * MTTKRP (Sec. 6.2, the first part of <MTTKRP,GEMM>), with the index names of
 * the C interface: A(i,l) = sum_{j,k} B(i,j,k) * C(j,l) * D(k,l).
 *
 * With B stored i -> j -> k in CSF, Algorithm 1 removes C: producer
 * T'(i,j,l) = sum_k B(i,j,k) D(k,l) (loops i, j, k, l), consumer
 * A(i,l) = sum_j T'(i,j,l) C(j,l) (loops i, j, l).  The common prefix is
 * {i, j}; below it l is shared, so the temporary is a vector over l, live for
 * one fiber (i,j).
 *
 * B: CSF (crd1[nslices] = i, pos2, crd2 = j, pos3, crd3 = k, vals), dims
 * d0 x d1 x d2.  C: d1 x L.  D: d2 x L.  A / A_abs: nsel x L for output rows
 * rows[0..nsel) (or 0..nsel-1); a row with no slice is zero.
 */
int oracle_mttkrp(int32_t d0, int32_t d1, int32_t d2, int32_t nslices, const int32_t *crd1,
                  const int32_t *pos2, const int32_t *crd2, const int32_t *pos3,
                  const int32_t *crd3, const float *vals, const float *C, const float *D,
                  int32_t L, int64_t nsel, const int32_t *rows, double *A, double *A_abs) {
  double *t = (double *)malloc(sizeof(double) * (size_t)(L > 0 ? L : 1));
  double *ta = (double *)malloc(sizeof(double) * (size_t)(L > 0 ? L : 1));
  if (!t || !ta) {
    free(t);
    free(ta);
    return -1;
  }
  int rc = 0;
  for (int64_t s = 0; s < nsel && rc == 0; ++s) {
    const int32_t i = rows ? rows[s] : (int32_t)s;
    double *a = A + s * L, *aa = A_abs + s * L;
    for (int32_t l = 0; l < L; ++l) {
      a[l] = 0.0;
      aa[l] = 0.0;
    }
    if (i < 0 || i >= d0) {
      rc = -1;
      break;
    }
    for (int32_t q = 0; q < nslices && rc == 0; ++q) {
      if (crd1[q] != i) continue;
      for (int32_t f = pos2[q]; f < pos2[q + 1] && rc == 0; ++f) {
        const int32_t j = crd2[f];
        if (j < 0 || j >= d1) {
          rc = -1;
          break;
        }
        /* producer: t(l) = sum_k B(i,j,k) D(k,l) */
        for (int32_t l = 0; l < L; ++l) {
          t[l] = 0.0;
          ta[l] = 0.0;
        }
        for (int32_t p = pos3[f]; p < pos3[f + 1]; ++p) {
          const int32_t k = crd3[p];
          if (k < 0 || k >= d2) {
            rc = -1;
            break;
          }
          const double b = (double)vals[p];
          for (int32_t l = 0; l < L; ++l) {
            const double d = (double)D[(int64_t)k * L + l];
            t[l] += b * d;
            ta[l] += fabs(b) * fabs(d);
          }
        }
        /* consumer: A(i,l) += t(l) C(j,l) */
        for (int32_t l = 0; l < L; ++l) {
          const double c = (double)C[(int64_t)j * L + l];
          a[l] += t[l] * c;
          aa[l] += ta[l] * fabs(c);
        }
      }
    }
  }
  free(t);
  free(ta);
  return rc;
}

/*
 * <SpTTM,SpTTM> (Sec. 6.2): A(i,j,m) = sum_{k,l} B(i,j,k) * C(k,l) * D(l,m),
 * A sparse in (i,j) and dense in m.
 *
 * Algorithm 1 removes D: producer T'(i,j,l) = sum_k B(i,j,k) C(k,l) (loops
 * i, j, k, l), consumer A(i,j,m) = sum_l T'(i,j,l) D(l,m) (loops i, j, l, m).
 * The common prefix is {i, j}; below it l is shared, so the temporary is a
 * vector over l per fiber, which gives the fused schedule's cost
 * O(nnz(B_IJK) L + nnz(B_IJ) L M) quoted in Sec. 6.2.
 *
 * Fibers evaluated: fibers[0..nsel) (or 0..nsel-1), each a position f in
 * B's fiber level (pos3[f]..pos3[f+1]).  C: d2 x L.  D: L x M.
 * A / A_abs: nsel x M.
 */
int oracle_spttm_ttm(int32_t nfibers, int32_t d2, const int32_t *pos3, const int32_t *crd3,
                     const float *vals, const float *C, int32_t L, const float *D, int32_t M,
                     int64_t nsel, const int32_t *fibers, double *A, double *A_abs) {
  double *t = (double *)malloc(sizeof(double) * (size_t)(L > 0 ? L : 1));
  double *ta = (double *)malloc(sizeof(double) * (size_t)(L > 0 ? L : 1));
  if (!t || !ta) {
    free(t);
    free(ta);
    return -1;
  }
  int rc = 0;
  for (int64_t s = 0; s < nsel && rc == 0; ++s) {
    const int32_t f = fibers ? fibers[s] : (int32_t)s;
    if (f < 0 || f >= nfibers || pos3[f] > pos3[f + 1]) {
      rc = -1;
      break;
    }
    /* producer: t(l) = sum_k B(i,j,k) C(k,l) */
    for (int32_t l = 0; l < L; ++l) {
      t[l] = 0.0;
      ta[l] = 0.0;
    }
    for (int32_t p = pos3[f]; p < pos3[f + 1]; ++p) {
      const int32_t k = crd3[p];
      if (k < 0 || k >= d2) {
        rc = -1;
        break;
      }
      const double b = (double)vals[p];
      for (int32_t l = 0; l < L; ++l) {
        const double c = (double)C[(int64_t)k * L + l];
        t[l] += b * c;
        ta[l] += fabs(b) * fabs(c);
      }
    }
    /* consumer: A(i,j,m) = sum_l t(l) D(l,m) */
    for (int32_t m = 0; m < M; ++m) {
      double acc = 0.0, acc_abs = 0.0;
      for (int32_t l = 0; l < L; ++l) {
        const double d = (double)D[(int64_t)l * M + m];
        acc += t[l] * d;
        acc_abs += ta[l] * fabs(d);
      }
      A[s * M + m] = acc;
      A_abs[s * M + m] = acc_abs;
    }
  }
  free(t);
  free(ta);
  return rc;
}

/*
 * Sparsity structure of the <SpTTM,SpTTM> output (Sec. 6.2 marks A_ijm
 * sparse, dense in m).  A(i,j,:) is stored for exactly the (i,j) that B
 * stores: the products with dense C and D create no new (i,j), and a fiber
 * whose values cancel to zero keeps its entry (no compaction).  A slice of B
 * that stores no fiber is kept as an empty slice of A.  This walks B's first
 * two levels in storage order and emits A's levels from them.
 *
 * Outputs: A_pos1[2], A_crd1[nslices], A_pos2[nslices+1], A_crd2[nfibers].
 * Returns the number of fibers of A, or -1 on malformed input.
 */
int64_t oracle_spttm_ttm_pattern(int32_t nslices, const int32_t *crd1, const int32_t *pos2,
                                 const int32_t *crd2, int32_t *A_pos1, int32_t *A_crd1,
                                 int32_t *A_pos2, int32_t *A_crd2) {
  int64_t nf = 0;
  A_pos2[0] = 0;
  for (int32_t q = 0; q < nslices; ++q) {
    if (pos2[q] > pos2[q + 1]) return -1;
    A_crd1[q] = crd1[q];
    for (int32_t f = pos2[q]; f < pos2[q + 1]; ++f) A_crd2[nf++] = crd2[f];
    A_pos2[q + 1] = (int32_t)nf;
  }
  A_pos1[0] = 0;
  A_pos1[1] = nslices;
  return nf;
}

/*
 * <SDDMM,SpMM,GEMM> (Sec. 6.2): A(i,m) = sum_{j,k,l} B(i,j) C(i,k) D(j,k) F(j,l) W(l,m)
 * -- the sampled products B(i,j) <C(i,:), D(j,:)>, a neighbour sum of F's rows
 * with those weights, and the product with W.
 *
 * Algorithm 1 applied recursively (Sec. 4.2 notes it can be reapplied to the
 * producer): removing W leaves producer P(i,l) = sum_j B(i,j) <C(i,:),D(j,:)>
 * F(j,l) (loops i, j, k, l) and consumer A(i,m) = sum_l P(i,l) W(l,m) (loops
 * i, l, m): common prefix {i}, temporary a vector over l per row.  The
 * producer is itself <SDDMM,SpMM>, whose temporary is a scalar per stored
 * (i,j).  So, per row i: for each stored j, y = B(i,j) <C(i,:), D(j,:)>,
 * t(l) += y F(j,l); then A(i,m) = sum_l t(l) W(l,m).
 *
 * B: nrows x ncols CSR.  C: nrows x K.  D: ncols x K.  F: ncols x L.
 * W: L x M.  Output rows as for oracle_spmm_gemm; A / A_abs are nsel x M.
 */
int oracle_sddmm_spmm_gemm(int32_t nrows, int32_t ncols, const int32_t *pos, const int32_t *crd,
                           const float *vals, const float *C, const float *D, int32_t K, const float *F,
                           int32_t L, const float *W, int32_t M, int64_t nsel, const int32_t *rows,
                           double *A, double *A_abs) {
  double *t = (double *)malloc(sizeof(double) * (size_t)(L > 0 ? L : 1));
  double *ta = (double *)malloc(sizeof(double) * (size_t)(L > 0 ? L : 1));
  if (!t || !ta) {
    free(t);
    free(ta);
    return -1;
  }
  int rc = 0;
  for (int64_t s = 0; s < nsel && rc == 0; ++s) {
    const int32_t i = rows ? rows[s] : (int32_t)s;
    if (!csr_row_ok(nrows, pos, i)) {
      rc = -1;
      break;
    }
    for (int32_t l = 0; l < L; ++l) {
      t[l] = 0.0;
      ta[l] = 0.0;
    }
    for (int32_t p = pos[i]; p < pos[i + 1]; ++p) {
      const int32_t j = crd[p];
      if (j < 0 || j >= ncols) {
        rc = -1;
        break;
      }
      const double b = (double)vals[p];
      /* innermost producer: the scalar y = B(i,j) sum_k C(i,k) D(j,k) */
      double y = 0.0, ya = 0.0;
      for (int32_t k = 0; k < K; ++k) {
        const double c = (double)C[(int64_t)i * K + k];
        const double d = (double)D[(int64_t)j * K + k];
        y += b * c * d;
        ya += fabs(b) * fabs(c) * fabs(d);
      }
      /* its consumer, the outer producer: t(l) += y F(j,l) */
      for (int32_t l = 0; l < L; ++l) {
        const double f = (double)F[(int64_t)j * L + l];
        t[l] += y * f;
        ta[l] += ya * fabs(f);
      }
    }
    /* outer consumer: A(i,m) = sum_l t(l) W(l,m) */
    for (int32_t m = 0; m < M; ++m) {
      double acc = 0.0, acc_abs = 0.0;
      for (int32_t l = 0; l < L; ++l) {
        const double w = (double)W[(int64_t)l * M + m];
        acc += t[l] * w;
        acc_abs += ta[l] * fabs(w);
      }
      A[s * M + m] = acc;
      A_abs[s * M + m] = acc_abs;
    }
  }
  free(t);
  free(ta);
  return rc;
}

/*
 * <MTTKRP,GEMM> (Sec. 6.2), with the index names of the C interface:
 * A(i,m) = sum_{j,k,l} B(i,j,k) C(j,l) D(k,l) E(l,m) -- MTTKRP followed by a
 * product with E (the paper prints A_im = sum B_ikl C_lj D_kj E_jm; its rank
 * index j is l here, as in oracle_mttkrp).
 *
 * Algorithm 1, applied twice: removing E leaves producer P(i,l) = MTTKRP and
 * consumer A(i,m) = sum_l P(i,l) E(l,m), common prefix {i}, temporary u(l)
 * per slice; the producer splits again as in oracle_mttkrp into t(l) per
 * fiber.  Per slice i: u(l) = sum_j t_j(l) C(j,l) with t_j(l) = sum_k
 * B(i,j,k) D(k,l); then A(i,m) = sum_l u(l) E(l,m).
 *
 * B: CSF (as oracle_mttkrp), dims d0 x d1 x d2.  C: d1 x L.  D: d2 x L.
 * E: L x M.  A / A_abs: nsel x M for output rows rows[0..nsel) (or
 * 0..nsel-1); a row with no slice is zero.
 */
int oracle_mttkrp_gemm(int32_t d0, int32_t d1, int32_t d2, int32_t nslices, const int32_t *crd1,
                       const int32_t *pos2, const int32_t *crd2, const int32_t *pos3,
                       const int32_t *crd3, const float *vals, const float *C, const float *D,
                       int32_t L, const float *E, int32_t M, int64_t nsel, const int32_t *rows,
                       double *A, double *A_abs) {
  double *t = (double *)malloc(sizeof(double) * (size_t)(L > 0 ? L : 1));
  double *ta = (double *)malloc(sizeof(double) * (size_t)(L > 0 ? L : 1));
  double *u = (double *)malloc(sizeof(double) * (size_t)(L > 0 ? L : 1));
  double *ua = (double *)malloc(sizeof(double) * (size_t)(L > 0 ? L : 1));
  if (!t || !ta || !u || !ua) {
    free(t);
    free(ta);
    free(u);
    free(ua);
    return -1;
  }
  int rc = 0;
  for (int64_t s = 0; s < nsel && rc == 0; ++s) {
    const int32_t i = rows ? rows[s] : (int32_t)s;
    if (i < 0 || i >= d0) {
      rc = -1;
      break;
    }
    for (int32_t l = 0; l < L; ++l) {
      u[l] = 0.0;
      ua[l] = 0.0;
    }
    for (int32_t q = 0; q < nslices && rc == 0; ++q) {
      if (crd1[q] != i) continue;
      for (int32_t f = pos2[q]; f < pos2[q + 1] && rc == 0; ++f) {
        const int32_t j = crd2[f];
        if (j < 0 || j >= d1) {
          rc = -1;
          break;
        }
        /* fiber producer: t(l) = sum_k B(i,j,k) D(k,l) */
        for (int32_t l = 0; l < L; ++l) {
          t[l] = 0.0;
          ta[l] = 0.0;
        }
        for (int32_t p = pos3[f]; p < pos3[f + 1]; ++p) {
          const int32_t k = crd3[p];
          if (k < 0 || k >= d2) {
            rc = -1;
            break;
          }
          const double b = (double)vals[p];
          for (int32_t l = 0; l < L; ++l) {
            const double d = (double)D[(int64_t)k * L + l];
            t[l] += b * d;
            ta[l] += fabs(b) * fabs(d);
          }
        }
        /* fiber consumer, slice producer: u(l) += t(l) C(j,l) */
        for (int32_t l = 0; l < L; ++l) {
          const double c = (double)C[(int64_t)j * L + l];
          u[l] += t[l] * c;
          ua[l] += ta[l] * fabs(c);
        }
      }
    }
    /* slice consumer: A(i,m) = sum_l u(l) E(l,m) */
    for (int32_t m = 0; m < M; ++m) {
      double acc = 0.0, acc_abs = 0.0;
      for (int32_t l = 0; l < L; ++l) {
        const double e = (double)E[(int64_t)l * M + m];
        acc += u[l] * e;
        acc_abs += ua[l] * fabs(e);
      }
      A[s * M + m] = acc;
      A_abs[s * M + m] = acc_abs;
    }
  }
  free(t);
  free(ta);
  free(u);
  free(ua);
  return rc;
}

/*
 * <SpMMH,GEMM> (Sec. 6.2): A(i,l) = sum_{k,j} B(i,k) C(k,j) D(k,j) E(j,l) -- a
 * sparse matrix times the Hadamard product of two dense matrices, then a
 * product with E.
 *
 * Algorithm 1 removes E: producer T'(i,j) = sum_k B(i,k) C(k,j) D(k,j) (loops
 * i, k, j), consumer A(i,l) = sum_j T'(i,j) E(j,l) (loops i, j, l).  Common
 * prefix {i}; below it j is shared, so the temporary is a vector over j per
 * row, as in <SpMM,GEMM>.
 *
 * B: nrows x ncols CSR (row i, column k).  C, D: ncols x J.  E: J x L.
 * Output rows as for oracle_spmm_gemm; A / A_abs are nsel x L.
 */
int oracle_spmmh_gemm(int32_t nrows, int32_t ncols, const int32_t *pos, const int32_t *crd,
                      const float *vals, const float *C, const float *D, int32_t J, const float *E,
                      int32_t L, int64_t nsel, const int32_t *rows, double *A, double *A_abs) {
  double *t = (double *)malloc(sizeof(double) * (size_t)(J > 0 ? J : 1));
  double *ta = (double *)malloc(sizeof(double) * (size_t)(J > 0 ? J : 1));
  if (!t || !ta) {
    free(t);
    free(ta);
    return -1;
  }
  int rc = 0;
  for (int64_t s = 0; s < nsel && rc == 0; ++s) {
    const int32_t i = rows ? rows[s] : (int32_t)s;
    if (!csr_row_ok(nrows, pos, i)) {
      rc = -1;
      break;
    }
    /* producer: t(j) = sum_k B(i,k) C(k,j) D(k,j) */
    for (int32_t j = 0; j < J; ++j) {
      t[j] = 0.0;
      ta[j] = 0.0;
    }
    for (int32_t p = pos[i]; p < pos[i + 1]; ++p) {
      const int32_t k = crd[p];
      if (k < 0 || k >= ncols) {
        rc = -1;
        break;
      }
      const double b = (double)vals[p];
      for (int32_t j = 0; j < J; ++j) {
        const double c = (double)C[(int64_t)k * J + j];
        const double d = (double)D[(int64_t)k * J + j];
        t[j] += b * c * d;
        ta[j] += fabs(b) * fabs(c) * fabs(d);
      }
    }
    /* consumer: A(i,l) = sum_j t(j) E(j,l) */
    for (int32_t l = 0; l < L; ++l) {
      double acc = 0.0, acc_abs = 0.0;
      for (int32_t j = 0; j < J; ++j) {
        const double e = (double)E[(int64_t)j * L + l];
        acc += t[j] * e;
        acc_abs += ta[j] * fabs(e);
      }
      A[s * L + l] = acc;
      A_abs[s * L + l] = acc_abs;
    }
  }
  free(t);
  free(ta);
  return rc;
}
