"""Checks that pin the oracle to facts outside itself.

Each ``check_*`` function runs one oracle (the real one, or a copy with a
planted mistake) against what the mathematics fixes, and returns the names of
the checks that fail:

* brute force -- B densified and the expression evaluated as the perfect loop
  nest over every index (the "TACO Original" schedule of Fig. 2c, Sec. 3.1.1),
  here by numpy.einsum in fp64 on tiny inputs with distinct dimension sizes, so
  that a transposed operand or a swapped index changes the result;
* exact integers -- small integer inputs, the dense definition evaluated with
  Python integers (exact), compared for equality;
* special cases that reduce to a library routine (scipy.sparse products),
  closed forms (a single nonzero), the magnitude companion's definition;
* linearity in every dense operand.

The fp64 tolerance is 1e-12 relative to the magnitude companion: far above
the rounding of a few hundred fp64 operations, far below any real mistake.
"""
from __future__ import annotations


import numpy as np
import scipy.sparse as sp

TOL = 1e-12


def _close(a, b, scale):
    a, b, scale = np.asarray(a), np.asarray(b), np.asarray(scale)
    return a.shape == b.shape and bool(np.all(np.abs(a - b) <= TOL * (np.abs(scale) + 1e-300)))


# --------------------------------------------------------------------------
# tiny random sparse inputs (test-side construction)

def rand_csr(rng, nrows, ncols, density, empty_rows=(), values="uniform"):
    mask = rng.random((nrows, ncols)) < density
    for r in empty_rows:
        mask[r, :] = False
    pos = np.zeros(nrows + 1, np.int32)
    crd, vals = [], []
    for i in range(nrows):
        cols = np.nonzero(mask[i])[0]
        crd.extend(cols.tolist())
        if values == "int":
            vals.extend(rng.integers(-3, 4, cols.shape[0]).tolist())
        else:
            vals.extend(rng.uniform(-1, 1, cols.shape[0]).tolist())
        pos[i + 1] = len(crd)
    return pos, np.array(crd, np.int32), np.array(vals, np.float32)


def csr_dense(nrows, ncols, pos, crd, vals):
    Bd = np.zeros((nrows, ncols))
    for i in range(nrows):
        for p in range(pos[i], pos[i + 1]):
            Bd[i, crd[p]] = vals[p]
    return Bd


def rand_csf(rng, dims, density, values="uniform", empty_slice_rows=()):
    d0, d1, d2 = dims
    mask = rng.random(dims) < density
    for i in empty_slice_rows:
        mask[i] = False
    crd1, pos2, crd2, pos3, crd3, vals = [], [0], [], [0], [], []
    for i in range(d0):
        if not mask[i].any():
            continue
        crd1.append(i)
        for j in range(d1):
            ks = np.nonzero(mask[i, j])[0]
            if ks.shape[0] == 0:
                continue
            crd2.append(j)
            crd3.extend(ks.tolist())
            if values == "int":
                vals.extend(rng.integers(-3, 4, ks.shape[0]).tolist())
            else:
                vals.extend(rng.uniform(-1, 1, ks.shape[0]).tolist())
            pos3.append(len(crd3))
        pos2.append(len(crd2))
    a = lambda x: np.array(x, np.int32)
    return a(crd1), a(pos2), a(crd2), a(pos3), a(crd3), np.array(vals, np.float32)


def csf_dense(dims, crd1, pos2, crd2, pos3, crd3, vals):
    Bd = np.zeros(dims)
    for q, i in enumerate(crd1):
        for f in range(pos2[q], pos2[q + 1]):
            for p in range(pos3[f], pos3[f + 1]):
                Bd[i, crd2[f], crd3[p]] = vals[p]
    return Bd


def f32(rng, shape, lo=-1.0, hi=1.0):
    return rng.uniform(lo, hi, shape).astype(np.float32)


def ints(rng, shape):
    return rng.integers(-3, 4, shape).astype(np.float32)


def dyadic(rng, shape):
    """Values m/1024 in [-1, 1]: a*X + b*Y stays exact in fp32 for dyadic a, b."""
    return (rng.integers(-1024, 1025, shape) / 1024.0).astype(np.float32)


def combo(a, X, b, Y):
    """a*X + b*Y formed in fp64; exact (and so unchanged by the fp32 cast) for dyadic inputs."""
    Z = a * X.astype(np.float64) + b * Y.astype(np.float64)
    Zf = Z.astype(np.float32)
    assert np.array_equal(Zf.astype(np.float64), Z), "linearity operands must combine exactly in fp32"
    return Zf


# --------------------------------------------------------------------------
# <SpMM,GEMM>

def check_spmm_gemm(orc, seed=1, square_kl=False):
    fails = []
    rng = np.random.default_rng(seed)
    nrows, ncols = 7, 9
    K, L = (5, 5) if square_kl else (5, 6)
    pos, crd, vals = rand_csr(rng, nrows, ncols, 0.4, empty_rows=(2,))
    C, D = f32(rng, (ncols, K)), f32(rng, (K, L))
    Bd = csr_dense(nrows, ncols, pos, crd, vals)
    A, Aa = orc.spmm_gemm(nrows, ncols, pos, crd, vals, C, D)
    ref = np.einsum("ij,jk,kl->il", Bd, C.astype(np.float64), D.astype(np.float64))
    ref_abs = np.einsum("ij,jk,kl->il", np.abs(Bd), np.abs(C.astype(np.float64)), np.abs(D.astype(np.float64)))
    if not _close(A, ref, ref_abs):
        fails.append("spmm_gemm brute force")
    if not _close(Aa, ref_abs, ref_abs):
        fails.append("spmm_gemm magnitude companion")
    if not np.all(A[2] == 0):
        fails.append("spmm_gemm empty row")
    # exact integers, dense definition in Python integers
    pos_i, crd_i, vals_i = rand_csr(rng, 4, 5, 0.5, values="int")
    Ci, Di = ints(rng, (5, 3)), ints(rng, (3, 3))
    Bi = csr_dense(4, 5, pos_i, crd_i, vals_i).astype(int).tolist()
    Cl, Dl = Ci.astype(int).tolist(), Di.astype(int).tolist()
    exact = [[sum(Bi[i][j] * Cl[j][k] * Dl[k][l] for j in range(5) for k in range(3)) for l in range(3)]
             for i in range(4)]
    Ai, _ = orc.spmm_gemm(4, 5, pos_i, crd_i, vals_i, Ci, Di)
    if not np.array_equal(Ai, np.array(exact, dtype=np.float64)):
        fails.append("spmm_gemm exact integers")
    # D = I reduces to SpMM (scipy CSR product)
    Kq = 6
    Cq = f32(rng, (ncols, Kq))
    Aq, Aqa = orc.spmm_gemm(nrows, ncols, pos, crd, vals, Cq, np.eye(Kq, dtype=np.float32))
    Bs = sp.csr_matrix((vals.astype(np.float64), crd, pos), shape=(nrows, ncols))
    if not _close(Aq, Bs @ Cq.astype(np.float64), Aqa):
        fails.append("spmm_gemm D=I is SpMM")
    # single nonzero B(i,j)=v: A[i,:] = v * C[j,:] @ D, all other rows zero
    p1 = np.array([0, 0, 0, 1, 1], np.int32)
    c1, v1 = np.array([4], np.int32), np.array([0.75], np.float32)
    A1, A1a = orc.spmm_gemm(4, ncols, p1, c1, v1, C, D)
    want = np.zeros((4, L)); want[2] = 0.75 * (C[4].astype(np.float64) @ D.astype(np.float64))
    if not _close(A1, want, A1a):
        fails.append("spmm_gemm single nonzero")
    # linearity in C and in D
    Cy, C2, Dy, D2 = dyadic(rng, (ncols, K)), dyadic(rng, (ncols, K)), dyadic(rng, (K, L)), dyadic(rng, (K, L))
    a, b = 0.5, -2.0
    A0, s0 = orc.spmm_gemm(nrows, ncols, pos, crd, vals, Cy, Dy)
    Aab, sab = orc.spmm_gemm(nrows, ncols, pos, crd, vals, combo(a, Cy, b, C2), Dy)
    A2, _ = orc.spmm_gemm(nrows, ncols, pos, crd, vals, C2, Dy)
    if not _close(Aab, a * A0 + b * A2, sab + s0):
        fails.append("spmm_gemm linear in C")
    Adb, sdb = orc.spmm_gemm(nrows, ncols, pos, crd, vals, Cy, combo(a, Dy, b, D2))
    A3, _ = orc.spmm_gemm(nrows, ncols, pos, crd, vals, Cy, D2)
    if not _close(Adb, a * A0 + b * A3, sdb + s0):
        fails.append("spmm_gemm linear in D")
    # row selection returns the same rows
    rows = np.array([6, 0, 2, 6], np.int32)
    As, _ = orc.spmm_gemm(nrows, ncols, pos, crd, vals, C, D, rows=rows)
    if not np.array_equal(As, A[rows]):
        fails.append("spmm_gemm row selection")
    return fails


# --------------------------------------------------------------------------
# <SDDMM,SpMM>: A(i,k) = sum_j B(i,j) (sum_l C(i,l) D(j,l)) E(j,k)

def check_sddmm_spmm(orc, seed=2):
    fails = []
    rng = np.random.default_rng(seed)
    n, L, K = 8, 5, 6
    pos, crd, vals = rand_csr(rng, n, n, 0.4, empty_rows=(3,))
    C, D, E = f32(rng, (n, L)), f32(rng, (n, L)), f32(rng, (n, K))
    Bd = csr_dense(n, n, pos, crd, vals)
    A, Aa = orc.sddmm_spmm(n, n, pos, crd, vals, C, D, E)
    C64, D64, E64 = (x.astype(np.float64) for x in (C, D, E))
    ref = np.einsum("ij,il,jl,jk->ik", Bd, C64, D64, E64)
    ref_abs = np.einsum("ij,il,jl,jk->ik", np.abs(Bd), np.abs(C64), np.abs(D64), np.abs(E64))
    if not _close(A, ref, ref_abs):
        fails.append("sddmm_spmm brute force")
    if not _close(Aa, ref_abs, ref_abs):
        fails.append("sddmm_spmm magnitude companion")
    # the separate schedule of Sec. 3.1.2: sampled product Y, then SpMM
    Y = Bd * (C64 @ D64.T)
    if not _close(A, Y @ E64, ref_abs):
        fails.append("sddmm_spmm equals SDDMM then SpMM")
    # exact integers on a rectangular B
    pos_i, crd_i, vals_i = rand_csr(rng, 4, 6, 0.5, values="int")
    Ci, Di, Ei = ints(rng, (4, 3)), ints(rng, (6, 3)), ints(rng, (6, 2))
    Bi = csr_dense(4, 6, pos_i, crd_i, vals_i).astype(int).tolist()
    Cl, Dl, El = (x.astype(int).tolist() for x in (Ci, Di, Ei))
    exact = [[sum(Bi[i][j] * sum(Cl[i][l] * Dl[j][l] for l in range(3)) * El[j][k] for j in range(6))
              for k in range(2)] for i in range(4)]
    Ai, _ = orc.sddmm_spmm(4, 6, pos_i, crd_i, vals_i, Ci, Di, Ei)
    if not np.array_equal(Ai, np.array(exact, dtype=np.float64)):
        fails.append("sddmm_spmm exact integers")
    # C(:,0) = D(:,0) = 1 and the rest 0: the scalar is B(i,j), so A = SpMM(B, E)
    Cu = np.zeros((n, L), np.float32); Cu[:, 0] = 1
    Du = np.zeros((n, L), np.float32); Du[:, 0] = 1
    Au, Aua = orc.sddmm_spmm(n, n, pos, crd, vals, Cu, Du, E)
    Bs = sp.csr_matrix((vals.astype(np.float64), crd, pos), shape=(n, n))
    if not _close(Au, Bs @ E64, Aua):
        fails.append("sddmm_spmm unit C,D is SpMM")
    # ... and with E = 1 every column is the row sum of B
    Ar, _ = orc.sddmm_spmm(n, n, pos, crd, vals, Cu, Du, np.ones((n, K), np.float32))
    rs = np.asarray(Bs.sum(axis=1)).ravel()
    if not _close(Ar, np.repeat(rs[:, None], K, axis=1), np.repeat(np.abs(Bd).sum(1)[:, None], K, 1)):
        fails.append("sddmm_spmm row sums")
    # linearity in E and in C (trilinear in C, D, E)
    Cy, C2, Ey, E2 = dyadic(rng, (n, L)), dyadic(rng, (n, L)), dyadic(rng, (n, K)), dyadic(rng, (n, K))
    a, b = 1.5, -0.25
    A0, s0 = orc.sddmm_spmm(n, n, pos, crd, vals, Cy, D, Ey)
    Ae, sae = orc.sddmm_spmm(n, n, pos, crd, vals, Cy, D, combo(a, Ey, b, E2))
    A2, _ = orc.sddmm_spmm(n, n, pos, crd, vals, Cy, D, E2)
    if not _close(Ae, a * A0 + b * A2, sae + s0):
        fails.append("sddmm_spmm linear in E")
    Ac, sac = orc.sddmm_spmm(n, n, pos, crd, vals, combo(a, Cy, b, C2), D, Ey)
    A3, _ = orc.sddmm_spmm(n, n, pos, crd, vals, C2, D, Ey)
    if not _close(Ac, a * A0 + b * A3, sac + s0):
        fails.append("sddmm_spmm linear in C")
    rows = np.array([7, 3, 0], np.int32)
    As, _ = orc.sddmm_spmm(n, n, pos, crd, vals, C, D, E, rows=rows)
    if not np.array_equal(As, A[rows]):
        fails.append("sddmm_spmm row selection")
    return fails


# --------------------------------------------------------------------------
# MTTKRP: A(i,l) = sum_{j,k} B(i,j,k) C(j,l) D(k,l)

def check_mttkrp(orc, seed=3):
    fails = []
    rng = np.random.default_rng(seed)
    dims, L = (6, 5, 7), 4
    csf = rand_csf(rng, dims, 0.25, empty_slice_rows=(1,))
    crd1, pos2, crd2, pos3, crd3, vals = csf
    C, D = f32(rng, (dims[1], L)), f32(rng, (dims[2], L))
    Bd = csf_dense(dims, *csf)
    A, Aa = orc.mttkrp(dims, *csf, C, D)
    C64, D64 = C.astype(np.float64), D.astype(np.float64)
    ref = np.einsum("ijk,jl,kl->il", Bd, C64, D64)
    ref_abs = np.einsum("ijk,jl,kl->il", np.abs(Bd), np.abs(C64), np.abs(D64))
    if not _close(A, ref, ref_abs):
        fails.append("mttkrp brute force")
    if not _close(Aa, ref_abs, ref_abs):
        fails.append("mttkrp magnitude companion")
    if not np.all(A[1] == 0):
        fails.append("mttkrp empty slice")
    # textbook matricised form: A = B_(1) (C kr D), column (j,k) -> j*d2 + k
    B1 = Bd.reshape(dims[0], dims[1] * dims[2])
    KR = (C64[:, None, :] * D64[None, :, :]).reshape(dims[1] * dims[2], L)
    if not _close(A, B1 @ KR, ref_abs):
        fails.append("mttkrp Khatri-Rao form")
    # L = 1, C = D = 1: each row is the sum of its slice's values
    A1, A1a = orc.mttkrp(dims, *csf, np.ones((dims[1], 1), np.float32), np.ones((dims[2], 1), np.float32))
    if not _close(A1[:, 0], Bd.sum(axis=(1, 2)), A1a[:, 0]):
        fails.append("mttkrp slice sums")
    # exact integers
    dims_i = (3, 4, 3)
    csf_i = rand_csf(rng, dims_i, 0.4, values="int")
    Ci, Di = ints(rng, (4, 2)), ints(rng, (3, 2))
    Bi = csf_dense(dims_i, *csf_i).astype(int).tolist()
    Cl, Dl = Ci.astype(int).tolist(), Di.astype(int).tolist()
    exact = [[sum(Bi[i][j][k] * Cl[j][l] * Dl[k][l] for j in range(4) for k in range(3)) for l in range(2)]
             for i in range(3)]
    Ai, _ = orc.mttkrp(dims_i, *csf_i, Ci, Di)
    if not np.array_equal(Ai, np.array(exact, dtype=np.float64)):
        fails.append("mttkrp exact integers")
    # linearity in C and D
    Cy, C2 = dyadic(rng, (dims[1], L)), dyadic(rng, (dims[1], L))
    Dy, D2 = dyadic(rng, (dims[2], L)), dyadic(rng, (dims[2], L))
    a, b = -1.25, 0.5
    A0, s0 = orc.mttkrp(dims, *csf, Cy, Dy)
    Acl, scl = orc.mttkrp(dims, *csf, combo(a, Cy, b, C2), Dy)
    A2, _ = orc.mttkrp(dims, *csf, C2, Dy)
    if not _close(Acl, a * A0 + b * A2, scl + s0):
        fails.append("mttkrp linear in C")
    Adl, sdl = orc.mttkrp(dims, *csf, Cy, combo(a, Dy, b, D2))
    A3, _ = orc.mttkrp(dims, *csf, Cy, D2)
    if not _close(Adl, a * A0 + b * A3, sdl + s0):
        fails.append("mttkrp linear in D")
    rows = np.array([5, 1, 0], np.int32)
    As, _ = orc.mttkrp(dims, *csf, C, D, rows=rows)
    if not np.array_equal(As, A[rows]):
        fails.append("mttkrp row selection")
    return fails


# --------------------------------------------------------------------------
# <SpTTM,SpTTM>: A(i,j,m) = sum_{k,l} B(i,j,k) C(k,l) D(l,m), A sparse in (i,j)

def check_spttm_ttm(orc, seed=4, square_lm=False):
    fails = []
    rng = np.random.default_rng(seed)
    dims = (4, 5, 6)
    L, M = (3, 3) if square_lm else (3, 4)
    csf = rand_csf(rng, dims, 0.3)
    crd1, pos2, crd2, pos3, crd3, vals = csf
    C, D = f32(rng, (dims[2], L)), f32(rng, (L, M))
    Bd = csf_dense(dims, *csf)
    A, Aa = orc.spttm_ttm(dims[2], pos3, crd3, vals, C, D)
    C64, D64 = C.astype(np.float64), D.astype(np.float64)
    ref_d = np.einsum("ijk,kl,lm->ijm", Bd, C64, D64)
    refa_d = np.einsum("ijk,kl,lm->ijm", np.abs(Bd), np.abs(C64), np.abs(D64))
    fiber_ij = [(crd1[q], crd2[f]) for q in range(crd1.shape[0]) for f in range(pos2[q], pos2[q + 1])]
    ref = np.array([ref_d[i, j] for i, j in fiber_ij])
    ref_abs = np.array([refa_d[i, j] for i, j in fiber_ij])
    if not _close(A, ref, ref_abs):
        fails.append("spttm_ttm brute force")
    if not _close(Aa, ref_abs, ref_abs):
        fails.append("spttm_ttm magnitude companion")
    # everything outside the stored (i,j) is zero in the dense result
    stored = np.zeros(dims[:2], bool)
    for i, j in fiber_ij:
        stored[i, j] = True
    if np.any(ref_d[~stored] != 0):
        fails.append("spttm_ttm output pattern covers the result")
    # re-associated schedule "separate2" (Sec. 6.2): B x_3 (C D)
    Bf = sp.csr_matrix((vals.astype(np.float64), crd3, pos3), shape=(len(fiber_ij), dims[2]))
    if not _close(A, Bf @ (C64 @ D64), ref_abs):
        fails.append("spttm_ttm re-association")
    # exact integers
    dims_i = (2, 3, 4)
    csf_i = rand_csf(rng, dims_i, 0.5, values="int")
    Ci, Di = ints(rng, (4, 2)), ints(rng, (2, 3))
    Bi = csf_dense(dims_i, *csf_i).astype(int).tolist()
    Cl, Dl = Ci.astype(int).tolist(), Di.astype(int).tolist()
    fij = [(csf_i[0][q], csf_i[2][f]) for q in range(csf_i[0].shape[0]) for f in range(csf_i[1][q], csf_i[1][q + 1])]
    exact = [[sum(Bi[i][j][k] * Cl[k][l] * Dl[l][m] for k in range(4) for l in range(2)) for m in range(3)]
             for i, j in fij]
    Ai, _ = orc.spttm_ttm(dims_i[2], csf_i[3], csf_i[4], csf_i[5], Ci, Di)
    if not np.array_equal(Ai, np.array(exact, dtype=np.float64)):
        fails.append("spttm_ttm exact integers")
    # linearity in C and D
    Cy, C2, Dy, D2 = dyadic(rng, (dims[2], L)), dyadic(rng, (dims[2], L)), dyadic(rng, (L, M)), dyadic(rng, (L, M))
    a, b = 0.75, -1.5
    A0, s0 = orc.spttm_ttm(dims[2], pos3, crd3, vals, Cy, Dy)
    Acl, scl = orc.spttm_ttm(dims[2], pos3, crd3, vals, combo(a, Cy, b, C2), Dy)
    A2, _ = orc.spttm_ttm(dims[2], pos3, crd3, vals, C2, Dy)
    if not _close(Acl, a * A0 + b * A2, scl + s0):
        fails.append("spttm_ttm linear in C")
    Adl, sdl = orc.spttm_ttm(dims[2], pos3, crd3, vals, Cy, combo(a, Dy, b, D2))
    A3, _ = orc.spttm_ttm(dims[2], pos3, crd3, vals, Cy, D2)
    if not _close(Adl, a * A0 + b * A3, sdl + s0):
        fails.append("spttm_ttm linear in D")
    fibers = np.array([len(fiber_ij) - 1, 0], np.int32)
    As, _ = orc.spttm_ttm(dims[2], pos3, crd3, vals, C, D, fibers=fibers)
    if not np.array_equal(As, A[fibers]):
        fails.append("spttm_ttm fiber selection")
    # output structure: levels rebuilt from the set of stored (i,j)
    p1, c1, p2, c2 = orc.spttm_ttm_pattern(crd1, pos2, crd2)
    ij_set = sorted({(int(i), int(j)) for i, j in fiber_ij})
    rebuilt = [(int(c1[q]), int(c2[f])) for q in range(c1.shape[0]) for f in range(p2[q], p2[q + 1])]
    if rebuilt != ij_set or list(p1) != [0, c1.shape[0]]:
        fails.append("spttm_ttm output pattern")
    return fails


# --------------------------------------------------------------------------
# <SDDMM,SpMM,GEMM>: A(i,m) = sum_{j,k,l} B(i,j) C(i,k) D(j,k) F(j,l) W(l,m)

def check_sddmm_spmm_gemm(orc, seed=5):
    fails = []
    rng = np.random.default_rng(seed)
    nrows, ncols, K, L, M = 7, 8, 3, 4, 5
    pos, crd, vals = rand_csr(rng, nrows, ncols, 0.4, empty_rows=(4,))
    C, D = f32(rng, (nrows, K)), f32(rng, (ncols, K))
    F, W = f32(rng, (ncols, L)), f32(rng, (L, M))
    Bd = csr_dense(nrows, ncols, pos, crd, vals)
    C64, D64, F64, W64 = (x.astype(np.float64) for x in (C, D, F, W))
    A, Aa = orc.sddmm_spmm_gemm(nrows, ncols, pos, crd, vals, C, D, F, W)
    ref = np.einsum("ij,ik,jk,jl,lm->im", Bd, C64, D64, F64, W64)
    ref_abs = np.einsum("ij,ik,jk,jl,lm->im", *(np.abs(x) for x in (Bd, C64, D64, F64, W64)))
    if not _close(A, ref, ref_abs):
        fails.append("sddmm_spmm_gemm brute force")
    if not _close(Aa, ref_abs, ref_abs):
        fails.append("sddmm_spmm_gemm magnitude companion")
    if not np.all(A[4] == 0):
        fails.append("sddmm_spmm_gemm empty row")
    # the paper's reading of the chain (Sec. 6.2): attention values on the
    # edges, the features times the weights, then the neighbour sum
    Y = Bd * (C64 @ D64.T)
    if not _close(A, Y @ (F64 @ W64), ref_abs):
        fails.append("sddmm_spmm_gemm equals SDDMM, then SpMM with F.W")
    # W = I: <SDDMM,SpMM>, here by scipy's sparse product of the sampled matrix
    Ai, Aia = orc.sddmm_spmm_gemm(nrows, ncols, pos, crd, vals, C, D, F, np.eye(L, dtype=np.float32))
    Ys = sp.csr_matrix((vals.astype(np.float64) * np.einsum("pk,pk->p", C64[np.repeat(np.arange(nrows), np.diff(pos))],
                                                             D64[crd]), crd, pos), shape=(nrows, ncols))
    if not _close(Ai, Ys @ F64, Aia):
        fails.append("sddmm_spmm_gemm W=I is SDDMM-SpMM")
    # exact integers
    pos_i, crd_i, vals_i = rand_csr(rng, 3, 4, 0.6, values="int")
    Ci, Di, Fi, Wi = ints(rng, (3, 2)), ints(rng, (4, 2)), ints(rng, (4, 3)), ints(rng, (3, 2))
    Bi = csr_dense(3, 4, pos_i, crd_i, vals_i).astype(int).tolist()
    Cl, Dl, Fl, Wl = (x.astype(int).tolist() for x in (Ci, Di, Fi, Wi))
    exact = [[sum(Bi[i][j] * Cl[i][k] * Dl[j][k] * Fl[j][l] * Wl[l][m]
                  for j in range(4) for k in range(2) for l in range(3)) for m in range(2)] for i in range(3)]
    Ae, _ = orc.sddmm_spmm_gemm(3, 4, pos_i, crd_i, vals_i, Ci, Di, Fi, Wi)
    if not np.array_equal(Ae, np.array(exact, dtype=np.float64)):
        fails.append("sddmm_spmm_gemm exact integers")
    # linearity in C, F and W
    Cy, C2 = dyadic(rng, (nrows, K)), dyadic(rng, (nrows, K))
    Fy, F2 = dyadic(rng, (ncols, L)), dyadic(rng, (ncols, L))
    Wy, W2 = dyadic(rng, (L, M)), dyadic(rng, (L, M))
    a, b = 0.5, -1.75
    run = lambda c, f, w: orc.sddmm_spmm_gemm(nrows, ncols, pos, crd, vals, c, D, f, w)
    A0, s0 = run(Cy, Fy, Wy)
    for name, args2, argsab in (("C", (C2, Fy, Wy), (combo(a, Cy, b, C2), Fy, Wy)),
                                ("F", (Cy, F2, Wy), (Cy, combo(a, Fy, b, F2), Wy)),
                                ("W", (Cy, Fy, W2), (Cy, Fy, combo(a, Wy, b, W2)))):
        Aab, sab = run(*argsab)
        A2, _ = run(*args2)
        if not _close(Aab, a * A0 + b * A2, sab + s0):
            fails.append(f"sddmm_spmm_gemm linear in {name}")
    rows = np.array([6, 4, 0], np.int32)
    As, _ = orc.sddmm_spmm_gemm(nrows, ncols, pos, crd, vals, C, D, F, W, rows=rows)
    if not np.array_equal(As, A[rows]):
        fails.append("sddmm_spmm_gemm row selection")
    return fails


# --------------------------------------------------------------------------
# <MTTKRP,GEMM>: A(i,m) = sum_{j,k,l} B(i,j,k) C(j,l) D(k,l) E(l,m)

def check_mttkrp_gemm(orc, seed=6):
    fails = []
    rng = np.random.default_rng(seed)
    dims, L, M = (6, 5, 7), 4, 3
    csf = rand_csf(rng, dims, 0.25, empty_slice_rows=(2,))
    C, D, E = f32(rng, (dims[1], L)), f32(rng, (dims[2], L)), f32(rng, (L, M))
    Bd = csf_dense(dims, *csf)
    C64, D64, E64 = (x.astype(np.float64) for x in (C, D, E))
    A, Aa = orc.mttkrp_gemm(dims, *csf, C, D, E)
    ref = np.einsum("ijk,jl,kl,lm->im", Bd, C64, D64, E64)
    ref_abs = np.einsum("ijk,jl,kl,lm->im", *(np.abs(x) for x in (Bd, C64, D64, E64)))
    if not _close(A, ref, ref_abs):
        fails.append("mttkrp_gemm brute force")
    if not _close(Aa, ref_abs, ref_abs):
        fails.append("mttkrp_gemm magnitude companion")
    if not np.all(A[2] == 0):
        fails.append("mttkrp_gemm empty slice")
    # matricised form B_(1) (C kr D) E
    B1 = Bd.reshape(dims[0], dims[1] * dims[2])
    KR = (C64[:, None, :] * D64[None, :, :]).reshape(dims[1] * dims[2], L)
    if not _close(A, B1 @ KR @ E64, ref_abs):
        fails.append("mttkrp_gemm Khatri-Rao form")
    # L = 1, C = D = 1: A(i,m) = (sum of slice i) * E(0,m)
    e1 = f32(rng, (1, M))
    A1, A1a = orc.mttkrp_gemm(dims, *csf, np.ones((dims[1], 1), np.float32), np.ones((dims[2], 1), np.float32), e1)
    if not _close(A1, np.outer(Bd.sum(axis=(1, 2)), e1[0].astype(np.float64)), A1a):
        fails.append("mttkrp_gemm slice sums")
    # exact integers
    dims_i = (3, 3, 4)
    csf_i = rand_csf(rng, dims_i, 0.4, values="int")
    Ci, Di, Ei = ints(rng, (3, 2)), ints(rng, (4, 2)), ints(rng, (2, 3))
    Bi = csf_dense(dims_i, *csf_i).astype(int).tolist()
    Cl, Dl, El = (x.astype(int).tolist() for x in (Ci, Di, Ei))
    exact = [[sum(Bi[i][j][k] * Cl[j][l] * Dl[k][l] * El[l][m] for j in range(3) for k in range(4) for l in range(2))
              for m in range(3)] for i in range(3)]
    Ae, _ = orc.mttkrp_gemm(dims_i, *csf_i, Ci, Di, Ei)
    if not np.array_equal(Ae, np.array(exact, dtype=np.float64)):
        fails.append("mttkrp_gemm exact integers")
    # linearity in C, D and E
    Cy, C2 = dyadic(rng, (dims[1], L)), dyadic(rng, (dims[1], L))
    Dy, D2 = dyadic(rng, (dims[2], L)), dyadic(rng, (dims[2], L))
    Ey, E2 = dyadic(rng, (L, M)), dyadic(rng, (L, M))
    a, b = -0.5, 2.0
    run = lambda c, d, e: orc.mttkrp_gemm(dims, *csf, c, d, e)
    A0, s0 = run(Cy, Dy, Ey)
    for name, args2, argsab in (("C", (C2, Dy, Ey), (combo(a, Cy, b, C2), Dy, Ey)),
                                ("D", (Cy, D2, Ey), (Cy, combo(a, Dy, b, D2), Ey)),
                                ("E", (Cy, Dy, E2), (Cy, Dy, combo(a, Ey, b, E2)))):
        Aab, sab = run(*argsab)
        A2, _ = run(*args2)
        if not _close(Aab, a * A0 + b * A2, sab + s0):
            fails.append(f"mttkrp_gemm linear in {name}")
    rows = np.array([5, 2, 0], np.int32)
    As, _ = orc.mttkrp_gemm(dims, *csf, C, D, E, rows=rows)
    if not np.array_equal(As, A[rows]):
        fails.append("mttkrp_gemm row selection")
    return fails


# --------------------------------------------------------------------------
# <SpMMH,GEMM>: A(i,l) = sum_{k,j} B(i,k) C(k,j) D(k,j) E(j,l)

def check_spmmh_gemm(orc, seed=7):
    fails = []
    rng = np.random.default_rng(seed)
    nrows, ncols, J, L = 6, 9, 4, 5
    pos, crd, vals = rand_csr(rng, nrows, ncols, 0.4, empty_rows=(1,))
    C, D, E = f32(rng, (ncols, J)), f32(rng, (ncols, J)), f32(rng, (J, L))
    Bd = csr_dense(nrows, ncols, pos, crd, vals)
    C64, D64, E64 = (x.astype(np.float64) for x in (C, D, E))
    A, Aa = orc.spmmh_gemm(nrows, ncols, pos, crd, vals, C, D, E)
    ref = np.einsum("ik,kj,kj,jl->il", Bd, C64, D64, E64)
    ref_abs = np.einsum("ik,kj,kj,jl->il", *(np.abs(x) for x in (Bd, C64, D64, E64)))
    if not _close(A, ref, ref_abs):
        fails.append("spmmh_gemm brute force")
    if not _close(Aa, ref_abs, ref_abs):
        fails.append("spmmh_gemm magnitude companion")
    if not np.all(A[1] == 0):
        fails.append("spmmh_gemm empty row")
    # D = 1: <SpMM,GEMM>, here by scipy's sparse product
    Bs = sp.csr_matrix((vals.astype(np.float64), crd, pos), shape=(nrows, ncols))
    A1, A1a = orc.spmmh_gemm(nrows, ncols, pos, crd, vals, C, np.ones_like(D), E)
    if not _close(A1, (Bs @ C64) @ E64, A1a):
        fails.append("spmmh_gemm D=1 is SpMM-GEMM")
    # single nonzero B(i,k)=v: A[i,:] = v (C[k,:] * D[k,:]) . E
    p1 = np.array([0, 0, 0, 0, 1], np.int32)
    c1, v1 = np.array([6], np.int32), np.array([-1.25], np.float32)
    As1, As1a = orc.spmmh_gemm(4, ncols, p1, c1, v1, C, D, E)
    want = np.zeros((4, L)); want[3] = -1.25 * ((C64[6] * D64[6]) @ E64)
    if not _close(As1, want, As1a):
        fails.append("spmmh_gemm single nonzero")
    # exact integers
    pos_i, crd_i, vals_i = rand_csr(rng, 3, 5, 0.5, values="int")
    Ci, Di, Ei = ints(rng, (5, 2)), ints(rng, (5, 2)), ints(rng, (2, 3))
    Bi = csr_dense(3, 5, pos_i, crd_i, vals_i).astype(int).tolist()
    Cl, Dl, El = (x.astype(int).tolist() for x in (Ci, Di, Ei))
    exact = [[sum(Bi[i][k] * Cl[k][j] * Dl[k][j] * El[j][l] for k in range(5) for j in range(2)) for l in range(3)]
             for i in range(3)]
    Ae, _ = orc.spmmh_gemm(3, 5, pos_i, crd_i, vals_i, Ci, Di, Ei)
    if not np.array_equal(Ae, np.array(exact, dtype=np.float64)):
        fails.append("spmmh_gemm exact integers")
    # linearity in C, D and E
    Cy, C2 = dyadic(rng, (ncols, J)), dyadic(rng, (ncols, J))
    Dy, D2 = dyadic(rng, (ncols, J)), dyadic(rng, (ncols, J))
    Ey, E2 = dyadic(rng, (J, L)), dyadic(rng, (J, L))
    a, b = 0.25, -3.0
    run = lambda c, d, e: orc.spmmh_gemm(nrows, ncols, pos, crd, vals, c, d, e)
    A0, s0 = run(Cy, Dy, Ey)
    for name, args2, argsab in (("C", (C2, Dy, Ey), (combo(a, Cy, b, C2), Dy, Ey)),
                                ("D", (Cy, D2, Ey), (Cy, combo(a, Dy, b, D2), Ey)),
                                ("E", (Cy, Dy, E2), (Cy, Dy, combo(a, Ey, b, E2)))):
        Aab, sab = run(*argsab)
        A2, _ = run(*args2)
        if not _close(Aab, a * A0 + b * A2, sab + s0):
            fails.append(f"spmmh_gemm linear in {name}")
    rows = np.array([5, 1, 2], np.int32)
    As, _ = orc.spmmh_gemm(nrows, ncols, pos, crd, vals, C, D, E, rows=rows)
    if not np.array_equal(As, A[rows]):
        fails.append("spmmh_gemm row selection")
    return fails


ALL_CHECKS = {
    "spmm_gemm": check_spmm_gemm,
    "sddmm_spmm": check_sddmm_spmm,
    "mttkrp": check_mttkrp,
    "spttm_ttm": check_spttm_ttm,
    "sddmm_spmm_gemm": check_sddmm_spmm_gemm,
    "mttkrp_gemm": check_mttkrp_gemm,
    "spmmh_gemm": check_spmmh_gemm,
}


def run_all(orc, seeds=(1, 2, 3)):
    fails = []
    for name, fn in ALL_CHECKS.items():
        for s in seeds:
            fails += [f"{f} (seed {s})" for f in fn(orc, seed=s)]
    fails += [f + " (K=L)" for f in check_spmm_gemm(orc, seed=9, square_kl=True)]
    fails += [f + " (L=M)" for f in check_spttm_ttm(orc, seed=9, square_lm=True)]
    return fails
