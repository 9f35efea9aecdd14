"""ORACLE -- test infrastructure, not part of the library.

ctypes binding of ``oracle.c``: the plain, single-threaded fp64 CPU evaluation
of the composite sparse expressions of SparseLNR's benchmarks (Sec. 6.2), in the loop
order that the paper's fusion-after-distribution transformation produces
(Sec. 4.2, Algorithm 1).  Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this package.  It never imports or
calls the CUDA library, and the CUDA library never uses it.

Every function returns ``(A, A_abs)`` as float64 arrays: the value and its
magnitude companion (the same loops on absolute values), used to bound the
error of any other summation order.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
SOURCE = os.path.join(_HERE, "oracle.c")
_BUILD = os.path.join(_HERE, "_build")
LIBRARY = os.path.join(_BUILD, "liboracle.so")
# Plain C with strict IEEE double arithmetic: no -ffast-math, no re-association.
CFLAGS = ["-std=c99", "-O2", "-fno-fast-math", "-ffp-contract=off", "-fPIC", "-shared"]


def compile_source(src: str, out: str) -> str:
    os.makedirs(os.path.dirname(out), exist_ok=True)
    tmp = out + f".tmp{os.getpid()}"
    subprocess.check_call(["gcc", *CFLAGS, src, "-o", tmp, "-lm"])
    os.replace(tmp, out)
    return out


def build(force: bool = False) -> str:
    if force or not os.path.exists(LIBRARY) or os.path.getmtime(LIBRARY) < os.path.getmtime(SOURCE):
        compile_source(SOURCE, LIBRARY)
    return LIBRARY


def _p(a):
    if a is None:
        return None
    assert a.flags["C_CONTIGUOUS"], "oracle inputs must be C-contiguous"
    return a.ctypes.data


def _i32(a):
    return np.ascontiguousarray(a, dtype=np.int32)


def _f32(a):
    return np.ascontiguousarray(a, dtype=np.float32)


class Oracle:
    """One loaded copy of the oracle library (tests may load planted-mistake copies)."""

    def __init__(self, path: str | None = None):
        self.path = path or build()
        lib = ctypes.CDLL(self.path)
        P, i32, i64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
        lib.oracle_spmm_gemm.argtypes = [i32, i32, P, P, P, P, i32, P, i32, i64, P, P, P]
        lib.oracle_spmm_gemm.restype = ctypes.c_int
        lib.oracle_sddmm_spmm.argtypes = [i32, i32, P, P, P, P, P, i32, P, i32, i64, P, P, P]
        lib.oracle_sddmm_spmm.restype = ctypes.c_int
        lib.oracle_mttkrp.argtypes = [i32, i32, i32, i32, P, P, P, P, P, P, P, P, i32, i64, P, P, P]
        lib.oracle_mttkrp.restype = ctypes.c_int
        lib.oracle_spttm_ttm.argtypes = [i32, i32, P, P, P, P, i32, P, i32, i64, P, P, P]
        lib.oracle_spttm_ttm.restype = ctypes.c_int
        lib.oracle_spttm_ttm_pattern.argtypes = [i32, P, P, P, P, P, P, P]
        lib.oracle_spttm_ttm_pattern.restype = ctypes.c_int64
        lib.oracle_sddmm_spmm_gemm.argtypes = [i32, i32, P, P, P, P, P, i32, P, i32, P, i32, i64, P, P, P]
        lib.oracle_sddmm_spmm_gemm.restype = ctypes.c_int
        lib.oracle_mttkrp_gemm.argtypes = [i32, i32, i32, i32, P, P, P, P, P, P, P, P, i32, P, i32, i64, P, P, P]
        lib.oracle_mttkrp_gemm.restype = ctypes.c_int
        lib.oracle_spmmh_gemm.argtypes = [i32, i32, P, P, P, P, P, i32, P, i32, i64, P, P, P]
        lib.oracle_spmmh_gemm.restype = ctypes.c_int
        self.lib = lib

    @staticmethod
    def _sel(rows, n):
        if rows is None:
            return None, n
        rows = _i32(rows)
        return rows, rows.shape[0]

    def spmm_gemm(self, nrows, ncols, pos, crd, vals, C, D, rows=None):
        """A(i,l) = sum_{j,k} B(i,j) C(j,k) D(k,l) for the selected rows i."""
        pos, crd, vals, C, D = _i32(pos), _i32(crd), _f32(vals), _f32(C), _f32(D)
        K, L = C.shape[1], D.shape[1]
        assert D.shape[0] == K and C.shape[0] == ncols
        sel, n = self._sel(rows, nrows)
        A = np.empty((n, L)); Aa = np.empty((n, L))
        rc = self.lib.oracle_spmm_gemm(nrows, ncols, _p(pos), _p(crd), _p(vals), _p(C), K, _p(D), L, n,
                                       _p(sel), _p(A), _p(Aa))
        if rc != 0:
            raise ValueError("oracle_spmm_gemm: malformed input")
        return A, Aa

    def sddmm_spmm(self, nrows, ncols, pos, crd, vals, C, D, E, rows=None):
        """A(i,k) = sum_j B(i,j) (sum_l C(i,l) D(j,l)) E(j,k) for the selected rows i."""
        pos, crd, vals, C, D, E = _i32(pos), _i32(crd), _f32(vals), _f32(C), _f32(D), _f32(E)
        L, K = C.shape[1], E.shape[1]
        assert C.shape[0] == nrows and D.shape == (ncols, L) and E.shape[0] == ncols
        sel, n = self._sel(rows, nrows)
        A = np.empty((n, K)); Aa = np.empty((n, K))
        rc = self.lib.oracle_sddmm_spmm(nrows, ncols, _p(pos), _p(crd), _p(vals), _p(C), _p(D), L, _p(E), K, n,
                                        _p(sel), _p(A), _p(Aa))
        if rc != 0:
            raise ValueError("oracle_sddmm_spmm: malformed input")
        return A, Aa

    def mttkrp(self, dims, crd1, pos2, crd2, pos3, crd3, vals, C, D, rows=None):
        """A(i,l) = sum_{j,k} B(i,j,k) C(j,l) D(k,l) for the selected rows i."""
        crd1, pos2, crd2, pos3, crd3 = map(_i32, (crd1, pos2, crd2, pos3, crd3))
        vals, C, D = _f32(vals), _f32(C), _f32(D)
        L = C.shape[1]
        assert C.shape[0] == dims[1] and D.shape == (dims[2], L)
        sel, n = self._sel(rows, dims[0])
        A = np.empty((n, L)); Aa = np.empty((n, L))
        rc = self.lib.oracle_mttkrp(dims[0], dims[1], dims[2], crd1.shape[0], _p(crd1), _p(pos2), _p(crd2),
                                    _p(pos3), _p(crd3), _p(vals), _p(C), _p(D), L, n, _p(sel), _p(A), _p(Aa))
        if rc != 0:
            raise ValueError("oracle_mttkrp: malformed input")
        return A, Aa

    def spttm_ttm(self, d2, pos3, crd3, vals, C, D, fibers=None):
        """A(i,j,m) = sum_{k,l} B(i,j,k) C(k,l) D(l,m) for the selected stored fibers (i,j)."""
        pos3, crd3, vals, C, D = _i32(pos3), _i32(crd3), _f32(vals), _f32(C), _f32(D)
        L, M = C.shape[1], D.shape[1]
        assert C.shape[0] == d2 and D.shape[0] == L
        nfib = pos3.shape[0] - 1
        sel, n = self._sel(fibers, nfib)
        A = np.empty((n, M)); Aa = np.empty((n, M))
        rc = self.lib.oracle_spttm_ttm(nfib, d2, _p(pos3), _p(crd3), _p(vals), _p(C), L, _p(D), M, n, _p(sel),
                                       _p(A), _p(Aa))
        if rc != 0:
            raise ValueError("oracle_spttm_ttm: malformed input")
        return A, Aa

    def spttm_ttm_pattern(self, crd1, pos2, crd2):
        """The two compressed levels (pos1, crd1, pos2, crd2) of the <SpTTM,SpTTM> output."""
        crd1, pos2, crd2 = _i32(crd1), _i32(pos2), _i32(crd2)
        ns, nf = crd1.shape[0], crd2.shape[0]
        p1 = np.empty(2, np.int32); c1 = np.empty(max(ns, 1), np.int32)
        p2 = np.empty(ns + 1, np.int32); c2 = np.empty(max(nf, 1), np.int32)
        got = self.lib.oracle_spttm_ttm_pattern(ns, _p(crd1), _p(pos2), _p(crd2), _p(p1), _p(c1), _p(p2), _p(c2))
        if got < 0:
            raise ValueError("oracle_spttm_ttm_pattern: malformed input")
        return p1, c1[:ns], p2, c2[:got]

    def sddmm_spmm_gemm(self, nrows, ncols, pos, crd, vals, C, D, F, W, rows=None):
        """A(i,m) = sum_{j,k,l} B(i,j) C(i,k) D(j,k) F(j,l) W(l,m) for the selected rows i."""
        pos, crd, vals = _i32(pos), _i32(crd), _f32(vals)
        C, D, F, W = _f32(C), _f32(D), _f32(F), _f32(W)
        K, L, M = C.shape[1], F.shape[1], W.shape[1]
        assert C.shape[0] == nrows and D.shape == (ncols, K) and F.shape[0] == ncols and W.shape[0] == L
        sel, n = self._sel(rows, nrows)
        A = np.empty((n, M)); Aa = np.empty((n, M))
        rc = self.lib.oracle_sddmm_spmm_gemm(nrows, ncols, _p(pos), _p(crd), _p(vals), _p(C), _p(D), K, _p(F), L,
                                             _p(W), M, n, _p(sel), _p(A), _p(Aa))
        if rc != 0:
            raise ValueError("oracle_sddmm_spmm_gemm: malformed input")
        return A, Aa

    def mttkrp_gemm(self, dims, crd1, pos2, crd2, pos3, crd3, vals, C, D, E, rows=None):
        """A(i,m) = sum_{j,k,l} B(i,j,k) C(j,l) D(k,l) E(l,m) for the selected rows i."""
        crd1, pos2, crd2, pos3, crd3 = map(_i32, (crd1, pos2, crd2, pos3, crd3))
        vals, C, D, E = _f32(vals), _f32(C), _f32(D), _f32(E)
        L, M = C.shape[1], E.shape[1]
        assert C.shape[0] == dims[1] and D.shape == (dims[2], L) and E.shape[0] == L
        sel, n = self._sel(rows, dims[0])
        A = np.empty((n, M)); Aa = np.empty((n, M))
        rc = self.lib.oracle_mttkrp_gemm(dims[0], dims[1], dims[2], crd1.shape[0], _p(crd1), _p(pos2), _p(crd2),
                                         _p(pos3), _p(crd3), _p(vals), _p(C), _p(D), L, _p(E), M, n, _p(sel),
                                         _p(A), _p(Aa))
        if rc != 0:
            raise ValueError("oracle_mttkrp_gemm: malformed input")
        return A, Aa

    def spmmh_gemm(self, nrows, ncols, pos, crd, vals, C, D, E, rows=None):
        """A(i,l) = sum_{k,j} B(i,k) C(k,j) D(k,j) E(j,l) for the selected rows i."""
        pos, crd, vals, C, D, E = _i32(pos), _i32(crd), _f32(vals), _f32(C), _f32(D), _f32(E)
        J, L = C.shape[1], E.shape[1]
        assert C.shape[0] == ncols and D.shape == C.shape and E.shape[0] == J
        sel, n = self._sel(rows, nrows)
        A = np.empty((n, L)); Aa = np.empty((n, L))
        rc = self.lib.oracle_spmmh_gemm(nrows, ncols, _p(pos), _p(crd), _p(vals), _p(C), _p(D), J, _p(E), L, n,
                                        _p(sel), _p(A), _p(Aa))
        if rc != 0:
            raise ValueError("oracle_spmmh_gemm: malformed input")
        return A, Aa

    # --- convenience on workloads.Workload objects ---------------------------------
    def run(self, w, rows=None):
        B, d = w.B, w.dense
        if w.op == "spmm_gemm":
            return self.spmm_gemm(B.nrows, B.ncols, B.pos, B.crd, B.vals, d["C"], d["D"], rows)
        if w.op == "sddmm_spmm":
            return self.sddmm_spmm(B.nrows, B.ncols, B.pos, B.crd, B.vals, d["C"], d["D"], d["E"], rows)
        if w.op == "mttkrp":
            return self.mttkrp(B.dims, B.crd1, B.pos2, B.crd2, B.pos3, B.crd3, B.vals, d["C"], d["D"], rows)
        if w.op == "spttm_ttm":
            return self.spttm_ttm(B.dims[2], B.pos3, B.crd3, B.vals, d["C"], d["D"], rows)
        if w.op == "sddmm_spmm_gemm":
            return self.sddmm_spmm_gemm(B.nrows, B.ncols, B.pos, B.crd, B.vals, d["C"], d["D"], d["F"], d["W"],
                                        rows)
        if w.op == "mttkrp_gemm":
            return self.mttkrp_gemm(B.dims, B.crd1, B.pos2, B.crd2, B.pos3, B.crd3, B.vals, d["C"], d["D"], d["E"],
                                    rows)
        if w.op == "spmmh_gemm":
            return self.spmmh_gemm(B.nrows, B.ncols, B.pos, B.crd, B.vals, d["C"], d["D"], d["E"], rows)
        raise ValueError(w.op)


_default = None
_lock = threading.Lock()


def get() -> Oracle:
    global _default
    with _lock:
        if _default is None:
            _default = Oracle()
    return _default
