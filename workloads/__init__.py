"""Seeded synthetic workloads shaped like the paper's benchmarks (Sec. 6.2).

This module only draws random numbers and builds sparse index structures
(CSR, CSF) plus dense fp32 operands; it holds none of the expressions'
arithmetic.  Both the CPU oracle and the CUDA library consume its output.
The C part (``gen.c``) is compiled on first use with the host ``gcc``.

The paper's own datasets (SuiteSparse, Network Repository, FROSTT, DARPA;
Table 1) are not available, so these synthetic inputs stand in for them:
R-MAT power-law graphs for the 2-D expressions, CSF tensors with Zipf slice
sizes or power-law fiber lengths for the 3-D ones.  Dense operands are random,
as they are in the paper (Sec. 6.1, "Dense tensors in kernels are randomly
generated").
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from dataclasses import dataclass, field

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "gen.c")
_BUILD = os.path.join(_HERE, "_build")
_SO = os.path.join(_BUILD, "libwl.so")
_lock = threading.Lock()
_lib = None

SEED_BASE = 0x51A4


def build(force: bool = False) -> str:
    """Compile gen.c into workloads/_build/libwl.so (gcc, no vendor flags)."""
    os.makedirs(_BUILD, exist_ok=True)
    if force or not os.path.exists(_SO) or os.path.getmtime(_SO) < os.path.getmtime(_SRC):
        tmp = _SO + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-std=gnu99", "-O2", "-fPIC", "-shared", _SRC, "-o", tmp, "-lm"])
        os.replace(tmp, _SO)
    return _SO


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            P = ctypes.c_void_p
            i32, i64, f32, f64 = ctypes.c_int32, ctypes.c_int64, ctypes.c_float, ctypes.c_double
            lib.wl_seed.argtypes = [P, ctypes.c_uint64]
            lib.wl_next.argtypes = [P]
            lib.wl_next.restype = ctypes.c_uint64
            lib.wl_fill_uniform.argtypes = [P, i64, f32, f32, P]
            lib.wl_fill_normal.argtypes = [P, i64, P]
            lib.wl_fill_const.argtypes = [i64, f32, P]
            lib.wl_uniform_csr.argtypes = [P, i32, i32, i32, P, P]
            lib.wl_uniform_csr.restype = i64
            lib.wl_rmat_csr.argtypes = [P, i32, i64, f64, f64, f64, P, P]
            lib.wl_rmat_csr.restype = i64
            lib.wl_zipf_slices_csf.argtypes = [P, i32, i32, i32, i64, f64, P, P, P, P, P, P]
            lib.wl_zipf_slices_csf.restype = i64
            lib.wl_powerlaw_fibers_csf.argtypes = [P, i32, i32, i32, i64, f64, i32, P, P, P, P, P, P]
            lib.wl_powerlaw_fibers_csf.restype = i64
            lib.wl_zipf_exponent_for_mean.argtypes = [i32, f64]
            lib.wl_zipf_exponent_for_mean.restype = f64
            _lib = lib
    return _lib


def _ptr(a: np.ndarray) -> int:
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data


class Rng:
    """xoshiro256** stream seeded through splitmix64 (state lives in C)."""

    def __init__(self, seed: int):
        self.state = (ctypes.c_uint64 * 4)()
        _load().wl_seed(ctypes.byref(self.state), ctypes.c_uint64(seed))

    @property
    def ref(self):
        return ctypes.byref(self.state)

    def next_u64(self) -> int:
        return int(_load().wl_next(self.ref))


def uniform(rng: Rng, shape, a: float, b: float) -> np.ndarray:
    out = np.empty(shape, dtype=np.float32)
    _load().wl_fill_uniform(rng.ref, out.size, a, b, _ptr(out))
    return out


def normal(rng: Rng, shape) -> np.ndarray:
    out = np.empty(shape, dtype=np.float32)
    _load().wl_fill_normal(rng.ref, out.size, _ptr(out))
    return out


def const(shape, v: float) -> np.ndarray:
    out = np.empty(shape, dtype=np.float32)
    _load().wl_fill_const(out.size, v, _ptr(out))
    return out


@dataclass
class CSR:
    """Compressed sparse rows: pos[nrows+1], crd[nnz] (sorted, unique per row), vals[nnz]."""

    nrows: int
    ncols: int
    pos: np.ndarray
    crd: np.ndarray
    vals: np.ndarray

    @property
    def nnz(self) -> int:
        return int(self.crd.shape[0])


@dataclass
class CSF3:
    """Compressed sparse fibers of a 3-tensor B(i,j,k), stored i -> j -> k.

    pos1 = [0, nslices]; crd1[nslices] (i); pos2[nslices+1]; crd2[nfibers] (j);
    pos3[nfibers+1]; crd3[nnz] (k); vals[nnz].
    """

    dims: tuple
    pos1: np.ndarray
    crd1: np.ndarray
    pos2: np.ndarray
    crd2: np.ndarray
    pos3: np.ndarray
    crd3: np.ndarray
    vals: np.ndarray

    @property
    def nnz(self) -> int:
        return int(self.crd3.shape[0])

    @property
    def nslices(self) -> int:
        return int(self.crd1.shape[0])

    @property
    def nfibers(self) -> int:
        return int(self.crd2.shape[0])


def uniform_csr_structure(rng: Rng, nrows: int, ncols: int, per_row: int):
    pos = np.empty(nrows + 1, dtype=np.int32)
    crd = np.empty(max(1, nrows * per_row), dtype=np.int32)
    nnz = _load().wl_uniform_csr(rng.ref, nrows, ncols, per_row, _ptr(pos), _ptr(crd))
    if nnz < 0:
        raise ValueError("wl_uniform_csr: bad arguments")
    return pos, crd[:nnz].copy()


def rmat_csr_structure(rng: Rng, n: int, nnz: int, a=0.57, b=0.19, c=0.19):
    pos = np.empty(n + 1, dtype=np.int32)
    crd = np.empty(max(1, nnz), dtype=np.int32)
    got = _load().wl_rmat_csr(rng.ref, n, nnz, a, b, c, _ptr(pos), _ptr(crd))
    if got < 0:
        raise ValueError("wl_rmat_csr: bad arguments")
    return pos, crd[:got].copy()


def _csf_buffers(d0: int, nnz: int):
    return (np.empty(d0, np.int32), np.empty(d0 + 1, np.int32), np.empty(max(1, nnz), np.int32),
            np.empty(nnz + 1, np.int32), np.empty(max(1, nnz), np.int32))


def _csf_from_buffers(dims, bufs, nslices, nfib, nnz, vals):
    crd1, pos2, crd2, pos3, crd3 = bufs
    return CSF3(dims=tuple(dims), pos1=np.array([0, nslices], np.int32), crd1=crd1[:nslices].copy(),
                pos2=pos2[:nslices + 1].copy(), crd2=crd2[:nfib].copy(), pos3=pos3[:nfib + 1].copy(),
                crd3=crd3[:nnz].copy(), vals=vals)


def zipf_slices_csf_structure(rng: Rng, dims, nnz: int, s: float):
    d0, d1, d2 = dims
    bufs = _csf_buffers(d0, nnz)
    ns = ctypes.c_int32(0)
    nfib = _load().wl_zipf_slices_csf(rng.ref, d0, d1, d2, nnz, s, *(_ptr(b) for b in bufs), ctypes.byref(ns))
    if nfib < 0:
        raise ValueError("wl_zipf_slices_csf: bad arguments")
    return bufs, ns.value, int(nfib)


def powerlaw_fibers_csf_structure(rng: Rng, dims, nnz: int, mean_len: float, max_len: int):
    d0, d1, d2 = dims
    bufs = _csf_buffers(d0, nnz)
    ns = ctypes.c_int32(0)
    nfib = _load().wl_powerlaw_fibers_csf(rng.ref, d0, d1, d2, nnz, mean_len, max_len,
                                          *(_ptr(b) for b in bufs), ctypes.byref(ns))
    if nfib < 0:
        raise ValueError("wl_powerlaw_fibers_csf: bad arguments")
    return bufs, ns.value, int(nfib)


def zipf_exponent_for_mean(max_len: int, mean_len: float) -> float:
    return float(_load().wl_zipf_exponent_for_mean(max_len, mean_len))


# --------------------------------------------------------------------------
# workload recipes (structure first, then values, then the dense operands)

@dataclass
class Workload:
    name: str
    op: str                       # spmm_gemm | sddmm_spmm | mttkrp | spttm_ttm | one of NEXT_OPS
    B: object                     # CSR or CSF3
    dense: dict = field(default_factory=dict)   # operand name -> fp32 array
    dims: dict = field(default_factory=dict)    # K, L, M as used by the op
    recipe: str = ""


def spmm_gemm_uniform(seed: int, nrows: int, ncols: int, per_row: int, K: int, L: int, name="spmm_gemm_uniform"):
    """<SpMM,GEMM> A = B.C.D with exactly per_row uniform columns per row; all values U[-1,1]."""
    r = Rng(seed)
    pos, crd = uniform_csr_structure(r, nrows, ncols, per_row)
    vals = uniform(r, crd.shape[0], -1.0, 1.0)
    C = uniform(r, (ncols, K), -1.0, 1.0)
    D = uniform(r, (K, L), -1.0, 1.0)
    return Workload(name, "spmm_gemm", CSR(nrows, ncols, pos, crd, vals), {"C": C, "D": D}, {"K": K, "L": L},
                    f"B {nrows}x{ncols} CSR, {per_row} distinct uniform cols/row, vals U[-1,1]; "
                    f"C {ncols}x{K}, D {K}x{L} U[-1,1]; seed {seed:#x}")


def spmm_gemm_rmat(seed: int, n: int, deg: int, K: int, L: int, name="spmm_gemm_rmat"):
    """<SpMM,GEMM> on an R-MAT(0.57,0.19,0.19) graph with n*deg distinct edges; vals U[-1,1]; C, D N(0,1)."""
    r = Rng(seed)
    pos, crd = rmat_csr_structure(r, n, n * deg)
    vals = uniform(r, crd.shape[0], -1.0, 1.0)
    C = normal(r, (n, K))
    D = normal(r, (K, L))
    return Workload(name, "spmm_gemm", CSR(n, n, pos, crd, vals), {"C": C, "D": D}, {"K": K, "L": L},
                    f"B {n}x{n} R-MAT(.57,.19,.19,.05), {n * deg} distinct edges, vals U[-1,1]; "
                    f"C {n}x{K}, D {K}x{L} N(0,1); seed {seed:#x}")


def sddmm_spmm_rmat(seed: int, n: int, deg: int, L: int, K: int, name="sddmm_spmm_rmat"):
    """<SDDMM,SpMM> A(i,k) = sum_j B(i,j) (sum_l C(i,l) D(j,l)) E(j,k); R-MAT, vals 1.0; C, D, E N(0,1)."""
    r = Rng(seed)
    pos, crd = rmat_csr_structure(r, n, n * deg)
    vals = const(crd.shape[0], 1.0)
    C = normal(r, (n, L))
    D = normal(r, (n, L))
    E = normal(r, (n, K))
    return Workload(name, "sddmm_spmm", CSR(n, n, pos, crd, vals), {"C": C, "D": D, "E": E}, {"K": K, "L": L},
                    f"B {n}x{n} R-MAT(.57,.19,.19,.05), {n * deg} distinct edges, vals 1.0; "
                    f"C,D {n}x{L}, E {n}x{K} N(0,1); seed {seed:#x}")


def mttkrp_zipf(seed: int, dims, nnz: int, s: float, L: int, name="mttkrp_zipf"):
    """MTTKRP A(i,l) = sum_{j,k} B(i,j,k) C(j,l) D(k,l); Zipf(s) slice sizes; vals U[0,1]; C, D U[-1,1]."""
    r = Rng(seed)
    bufs, ns, nfib = zipf_slices_csf_structure(r, dims, nnz, s)
    vals = uniform(r, nnz, 0.0, 1.0)
    B = _csf_from_buffers(dims, bufs, ns, nfib, nnz, vals)
    C = uniform(r, (dims[1], L), -1.0, 1.0)
    D = uniform(r, (dims[2], L), -1.0, 1.0)
    return Workload(name, "mttkrp", B, {"C": C, "D": D}, {"L": L},
                    f"B {dims[0]}x{dims[1]}x{dims[2]} CSF, {nnz} nnz, Zipf({s}) slice sizes, vals U[0,1]; "
                    f"C {dims[1]}x{L}, D {dims[2]}x{L} U[-1,1]; seed {seed:#x}")


def spttm_ttm_powerlaw(seed: int, dims, nnz: int, mean_len: float, max_len: int, L: int, M: int,
                       name="spttm_ttm_powerlaw"):
    """<SpTTM,SpTTM> A(i,j,m) = sum_{k,l} B(i,j,k) C(k,l) D(l,m); power-law fiber lengths; vals U[-1,1]; C, D N(0,1)."""
    r = Rng(seed)
    bufs, ns, nfib = powerlaw_fibers_csf_structure(r, dims, nnz, mean_len, max_len)
    vals = uniform(r, nnz, -1.0, 1.0)
    B = _csf_from_buffers(dims, bufs, ns, nfib, nnz, vals)
    C = normal(r, (dims[2], L))
    D = normal(r, (L, M))
    return Workload(name, "spttm_ttm", B, {"C": C, "D": D}, {"L": L, "M": M},
                    f"B {dims[0]}x{dims[1]}x{dims[2]} CSF, {nnz} nnz, fiber lengths truncated Zipf on "
                    f"[1,{max_len}] with mean {mean_len}, vals U[-1,1]; C {dims[2]}x{L}, D {L}x{M} N(0,1); "
                    f"seed {seed:#x}")


def sddmm_spmm_gemm_rmat(seed: int, n: int, deg: int, K: int, L: int, M: int, name="sddmm_spmm_gemm_rmat"):
    """<SDDMM,SpMM,GEMM> A(i,m) = sum B(i,j) C(i,k) D(j,k) F(j,l) W(l,m); R-MAT, vals 1.0; C, D, F, W N(0,1)."""
    r = Rng(seed)
    pos, crd = rmat_csr_structure(r, n, n * deg)
    vals = const(crd.shape[0], 1.0)
    C = normal(r, (n, K))
    D = normal(r, (n, K))
    F = normal(r, (n, L))
    W = normal(r, (L, M))
    return Workload(name, "sddmm_spmm_gemm", CSR(n, n, pos, crd, vals), {"C": C, "D": D, "F": F, "W": W},
                    {"K": K, "L": L, "M": M},
                    f"B {n}x{n} R-MAT(.57,.19,.19,.05), {n * deg} distinct edges, vals 1.0; "
                    f"C,D {n}x{K}, F {n}x{L}, W {L}x{M} N(0,1); seed {seed:#x}")


def mttkrp_gemm_zipf(seed: int, dims, nnz: int, s: float, L: int, M: int, name="mttkrp_gemm_zipf"):
    """<MTTKRP,GEMM> A(i,m) = sum B(i,j,k) C(j,l) D(k,l) E(l,m); Zipf(s) slices; vals U[0,1]; C, D, E U[-1,1]."""
    r = Rng(seed)
    bufs, ns, nfib = zipf_slices_csf_structure(r, dims, nnz, s)
    vals = uniform(r, nnz, 0.0, 1.0)
    B = _csf_from_buffers(dims, bufs, ns, nfib, nnz, vals)
    C = uniform(r, (dims[1], L), -1.0, 1.0)
    D = uniform(r, (dims[2], L), -1.0, 1.0)
    E = uniform(r, (L, M), -1.0, 1.0)
    return Workload(name, "mttkrp_gemm", B, {"C": C, "D": D, "E": E}, {"L": L, "M": M},
                    f"B {dims[0]}x{dims[1]}x{dims[2]} CSF, {nnz} nnz, Zipf({s}) slice sizes, vals U[0,1]; "
                    f"C {dims[1]}x{L}, D {dims[2]}x{L}, E {L}x{M} U[-1,1]; seed {seed:#x}")


def spmmh_gemm_rmat(seed: int, n: int, deg: int, J: int, L: int, name="spmmh_gemm_rmat"):
    """<SpMMH,GEMM> A(i,l) = sum B(i,k) C(k,j) D(k,j) E(j,l); R-MAT, vals U[-1,1]; C, D, E N(0,1)."""
    r = Rng(seed)
    pos, crd = rmat_csr_structure(r, n, n * deg)
    vals = uniform(r, crd.shape[0], -1.0, 1.0)
    C = normal(r, (n, J))
    D = normal(r, (n, J))
    E = normal(r, (J, L))
    return Workload(name, "spmmh_gemm", CSR(n, n, pos, crd, vals), {"C": C, "D": D, "E": E}, {"J": J, "L": L},
                    f"B {n}x{n} R-MAT(.57,.19,.19,.05), {n * deg} distinct edges, vals U[-1,1]; "
                    f"C,D {n}x{J}, E {J}x{L} N(0,1); seed {seed:#x}")


# The five benchmark workloads at full size (index = position in the benchmark
# list).  `scale` < 1 shrinks the row count (R-MAT) or the nonzero count (CSF)
# with the same recipe, for profiling captures on smaller cases.
def full(index: int, scale: float = 1.0) -> Workload:
    seed = SEED_BASE + index
    tag = "" if scale == 1.0 else f"_x{scale:g}"
    if index == 0:
        return spmm_gemm_uniform(seed, 1024, 1024, 10, 32, 32, name="spmm_gemm_1k_k32")
    if index == 1:
        return sddmm_spmm_rmat(seed, int(100_000 * scale), 20, 64, 64, name="sddmm_spmm_rmat100k_d20_64" + tag)
    if index == 2:
        return spmm_gemm_rmat(seed, int((1 << 20) * scale), 16, 128, 128, name="spmm_gemm_rmat1m_d16_k128" + tag)
    if index == 3:
        return mttkrp_zipf(seed, (10_000, 10_000, 10_000), int(10_000_000 * scale), 1.2, 32,
                           name="mttkrp_zipf10k_10m_l32" + tag)
    if index == 4:
        return spttm_ttm_powerlaw(seed, (5_000, 5_000, 5_000), int(20_000_000 * scale), 8.0, 5_000, 64, 64,
                                  name="spttm_ttm_powerlaw5k_20m_64" + tag)
    raise IndexError(index)


# Reduced versions with the same structure recipe: several tiles, heavy rows,
# ragged tails, and sizes the oracle finishes in well under a second.
def small(index: int, seed_offset: int = 100) -> Workload:
    seed = SEED_BASE + index + seed_offset
    if index == 0:
        return spmm_gemm_uniform(seed, 1024, 1024, 10, 32, 32, name="spmm_gemm_1k_k32")
    if index == 1:
        return sddmm_spmm_rmat(seed, 3001, 20, 64, 64, name="sddmm_spmm_rmat3001")
    if index == 2:
        return spmm_gemm_rmat(seed, 5003, 16, 128, 128, name="spmm_gemm_rmat5003")
    if index == 3:
        return mttkrp_zipf(seed, (300, 200, 400), 60_000, 1.2, 32, name="mttkrp_zipf300")
    if index == 4:
        return spttm_ttm_powerlaw(seed, (150, 170, 400), 40_000, 8.0, 400, 64, 64, name="spttm_ttm_powerlaw400")
    raise IndexError(index)


# The further expressions of Sec. 6.2 (<SDDMM,SpMM,GEMM> with k,l,m = 64,64,64;
# <MTTKRP,GEMM> with rank 32 and m = 64; <SpMMH,GEMM> with j,l = 128,128), on
# the structures of the benchmark workloads above: index 0, 1, 2.
NEXT_OPS = ("sddmm_spmm_gemm", "mttkrp_gemm", "spmmh_gemm")


def next_full(index: int, scale: float = 1.0) -> Workload:
    seed = SEED_BASE + 5 + index
    tag = "" if scale == 1.0 else f"_x{scale:g}"
    if index == 0:
        return sddmm_spmm_gemm_rmat(seed, int(100_000 * scale), 20, 64, 64, 64,
                                    name="sddmm_spmm_gemm_rmat100k_d20_64" + tag)
    if index == 1:
        return mttkrp_gemm_zipf(seed, (10_000, 10_000, 10_000), int(10_000_000 * scale), 1.2, 32, 64,
                                name="mttkrp_gemm_zipf10k_10m_32_64" + tag)
    if index == 2:
        return spmmh_gemm_rmat(seed, int((1 << 20) * scale), 16, 128, 128, name="spmmh_gemm_rmat1m_d16_128" + tag)
    raise IndexError(index)


def next_small(index: int, seed_offset: int = 100) -> Workload:
    seed = SEED_BASE + 5 + index + seed_offset
    if index == 0:
        return sddmm_spmm_gemm_rmat(seed, 3001, 20, 64, 64, 64, name="sddmm_spmm_gemm_rmat3001")
    if index == 1:
        return mttkrp_gemm_zipf(seed, (300, 200, 400), 60_000, 1.2, 32, 64, name="mttkrp_gemm_zipf300")
    if index == 2:
        return spmmh_gemm_rmat(seed, 5003, 16, 128, 128, name="spmmh_gemm_rmat5003")
    raise IndexError(index)
