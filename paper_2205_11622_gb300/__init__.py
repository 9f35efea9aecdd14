"""Thin Python binding of libslnr (include/slnr.h): fused composite sparse
tensor expressions on one GB300 (sm_103a).

The expressions and their fused schedules come from SparseLNR (Dias et al.,
ICS'22), Sec. 6.2; every step runs in the library's CUDA kernels.  This module
only marshals arguments: it turns torch CUDA tensors into the C structures
and device pointers of the ABI, allocates the caller-side workspace, passes
the current CUDA stream and raises on a non-zero status.  There is no CPU
path: if the library is missing or no GPU is present the calls raise.

Low-level entry points carry the C names (``slnr_spmm_gemm`` ...) and take
ctypes structures and raw device pointers; the snake-case wrappers
(``spmm_gemm`` ...) take torch tensors.
"""
from __future__ import annotations

import ctypes
import os
import threading
from dataclasses import dataclass

from . import build as _build

LIBRARY = _build.LIBRARY

FUSED, UNFUSED = 0, 1
STATUS = {0: "SLNR_OK", 1: "SLNR_ERR_NULL", 2: "SLNR_ERR_SHAPE", 3: "SLNR_ERR_INDEX", 4: "SLNR_ERR_WORKSPACE",
          5: "SLNR_ERR_UNSUPPORTED", 6: "SLNR_ERR_CUDA", 7: "SLNR_ERR_TIMEOUT"}


class SlnrError(RuntimeError):
    def __init__(self, status: int, where: str, detail: str):
        super().__init__(f"{where}: {STATUS.get(status, status)}: {detail}")
        self.status = status


class slnr_csr(ctypes.Structure):
    _fields_ = [("nrows", ctypes.c_int32), ("ncols", ctypes.c_int32), ("nnz", ctypes.c_int64),
                ("pos", ctypes.c_void_p), ("crd", ctypes.c_void_p), ("vals", ctypes.c_void_p)]


class slnr_csf3(ctypes.Structure):
    _fields_ = [("dim", ctypes.c_int32 * 3), ("nnz", ctypes.c_int64), ("nslices", ctypes.c_int32),
                ("nfibers", ctypes.c_int32), ("pos1", ctypes.c_void_p), ("crd1", ctypes.c_void_p),
                ("pos2", ctypes.c_void_p), ("crd2", ctypes.c_void_p), ("pos3", ctypes.c_void_p),
                ("crd3", ctypes.c_void_p), ("vals", ctypes.c_void_p)]


class slnr_opts(ctypes.Structure):
    _fields_ = [("variant", ctypes.c_int32), ("allow_tf32", ctypes.c_int32), ("validate", ctypes.c_int32),
                ("reserved", ctypes.c_int32), ("stream", ctypes.c_void_p), ("workspace", ctypes.c_void_p),
                ("workspace_bytes", ctypes.c_size_t)]


# name -> (argtypes, restype) of every symbol declared in include/slnr.h
_P, _I32, _SZ = ctypes.c_void_p, ctypes.c_int32, ctypes.POINTER(ctypes.c_size_t)
_CSR, _CSF, _OPT = ctypes.POINTER(slnr_csr), ctypes.POINTER(slnr_csf3), ctypes.POINTER(slnr_opts)
SIGNATURES = {
    "slnr_spmm_gemm_workspace": ([_CSR, _I32, _I32, _OPT, _SZ], ctypes.c_int),
    "slnr_sddmm_spmm_workspace": ([_CSR, _I32, _I32, _OPT, _SZ], ctypes.c_int),
    "slnr_mttkrp_workspace": ([_CSF, _I32, _OPT, _SZ], ctypes.c_int),
    "slnr_spttm_ttm_workspace": ([_CSF, _I32, _I32, _OPT, _SZ], ctypes.c_int),
    "slnr_sddmm_spmm_gemm_workspace": ([_CSR, _I32, _I32, _I32, _OPT, _SZ], ctypes.c_int),
    "slnr_mttkrp_gemm_workspace": ([_CSF, _I32, _I32, _OPT, _SZ], ctypes.c_int),
    "slnr_spmmh_gemm_workspace": ([_CSR, _I32, _I32, _OPT, _SZ], ctypes.c_int),
    "slnr_spmm_gemm": ([_CSR, _P, _I32, _P, _I32, _P, _OPT], ctypes.c_int),
    "slnr_spmm_gemm_original": ([_CSR, _P, _I32, _P, _I32, _P, _P], ctypes.c_int),
    "slnr_sddmm_spmm": ([_CSR, _P, _P, _I32, _P, _I32, _P, _OPT], ctypes.c_int),
    "slnr_mttkrp": ([_CSF, _P, _P, _I32, _P, _OPT], ctypes.c_int),
    "slnr_spttm_ttm": ([_CSF, _P, _I32, _P, _I32, _P, _P, _P, _P, _P, _OPT], ctypes.c_int),
    "slnr_sddmm_spmm_gemm": ([_CSR, _P, _P, _I32, _P, _I32, _P, _I32, _P, _OPT], ctypes.c_int),
    "slnr_mttkrp_gemm": ([_CSF, _P, _P, _I32, _P, _I32, _P, _OPT], ctypes.c_int),
    "slnr_spmmh_gemm": ([_CSR, _P, _P, _I32, _P, _I32, _P, _OPT], ctypes.c_int),
    "slnr_sddmm_spmm_noalloc": ([_CSR, _P, _P, _I32, _P, _I32, _P, _P], ctypes.c_int),
    "slnr_set_wait_limit": ([ctypes.c_int64], ctypes.c_int),
    "slnr_peak_ffma": ([_P, ctypes.POINTER(ctypes.c_double)], ctypes.c_int),
    "slnr_peak_tf32": ([_P, ctypes.POINTER(ctypes.c_double)], ctypes.c_int),
    "slnr_timing_launches": ([], ctypes.c_int32),
    "slnr_peak_gather": ([_P, ctypes.c_int64, ctypes.c_int, _P, ctypes.POINTER(ctypes.c_double)], ctypes.c_int),
    "slnr_timing_enable": ([_I32], ctypes.c_int),
    "slnr_timing_count": ([], ctypes.c_int32),
    "slnr_timing_get": ([_I32, ctypes.POINTER(ctypes.c_char_p), ctypes.POINTER(ctypes.c_float)], ctypes.c_int),
    "slnr_status_string": ([ctypes.c_int], ctypes.c_char_p),
    "slnr_last_error": ([], ctypes.c_char_p),
    "slnr_version": ([], ctypes.c_char_p),
}

_lib = None
_lock = threading.Lock()


def build(force: bool = False) -> str:
    """Compile libslnr.so for sm_103a (nvcc); returns its path."""
    return _build.build(force=force)


def lib():
    """The loaded libslnr.so.  Raises if it has not been built: there is no fallback."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(LIBRARY):
                raise RuntimeError(f"libslnr.so is not built ({LIBRARY}); call paper_2205_11622_gb300.build()")
            l = ctypes.CDLL(LIBRARY)
            for name, (args, res) in SIGNATURES.items():
                fn = getattr(l, name)
                fn.argtypes = args
                fn.restype = res
            _lib = l
    return _lib


def last_error() -> str:
    return lib().slnr_last_error().decode()


def _check(status: int, where: str):
    if status != 0:
        raise SlnrError(status, where, last_error())


def timing_enable(on: bool = True):
    """Record CUDA events between the library's launches on this thread (slnr_timing_enable)."""
    _check(lib().slnr_timing_enable(int(bool(on))), "slnr_timing_enable")


def peaks(stream=None, gather_width=None):
    """{"ffma_tflops", "tf32_tflops"}: the compute peaks measured by the library's own kernels.

    With gather_width (a power of two in [4, 128]) also "l2_gather_gbs" and
    "hbm_gather_gbs": the rate of whole-row gathers of that width from a
    table of a quarter of L2 and from one of 2 GB (slnr_peak_gather)."""
    torch = _torch()
    st = stream or torch.cuda.current_stream()
    s = ctypes.c_void_p(st.cuda_stream)
    out = {}
    for key, fn in (("ffma_tflops", "slnr_peak_ffma"), ("tf32_tflops", "slnr_peak_tf32")):
        v = ctypes.c_double(0.0)
        _check(getattr(lib(), fn)(s, ctypes.byref(v)), fn)
        out[key] = v.value
    if gather_width is not None:
        dev = torch.device("cuda", torch.cuda.current_device())
        l2 = torch.cuda.get_device_properties(dev).L2_cache_size
        for key, nbytes in (("l2_gather_gbs", l2 // 4), ("hbm_gather_gbs", 2 << 30)):
            rows = nbytes // (4 * gather_width)
            with torch.cuda.stream(st):
                table = torch.zeros((rows, gather_width), dtype=torch.float32, device=dev)
            v = ctypes.c_double(0.0)
            _check(lib().slnr_peak_gather(ctypes.c_void_p(table.data_ptr()), rows, gather_width, s,
                                          ctypes.byref(v)), "slnr_peak_gather")
            out[key] = v.value
            del table
    return out


def timing_launches():
    """Kernel launches of the calling thread's last call (slnr_timing_launches)."""
    return int(lib().slnr_timing_launches())


def timing_read():
    """[(kernel name, device ms)] of the calling thread's last call; waits for that call."""
    out = []
    for i in range(lib().slnr_timing_count()):
        name, ms = ctypes.c_char_p(), ctypes.c_float()
        _check(lib().slnr_timing_get(i, ctypes.byref(name), ctypes.byref(ms)), "slnr_timing_get")
        out.append((name.value.decode(), float(ms.value)))
    return out


# ---- low-level entry points (C names, raw pointers) -----------------------------------

def slnr_spmm_gemm(B, C, K, D, L, A, opts):
    return lib().slnr_spmm_gemm(ctypes.byref(B), C, K, D, L, A, ctypes.byref(opts))


def slnr_sddmm_spmm(B, C, D, L, E, K, A, opts):
    return lib().slnr_sddmm_spmm(ctypes.byref(B), C, D, L, E, K, A, ctypes.byref(opts))


def slnr_mttkrp(B, C, D, L, A, opts):
    return lib().slnr_mttkrp(ctypes.byref(B), C, D, L, A, ctypes.byref(opts))


def slnr_spttm_ttm(B, C, L, D, M, A_pos1, A_crd1, A_pos2, A_crd2, A_vals, opts):
    return lib().slnr_spttm_ttm(ctypes.byref(B), C, L, D, M, A_pos1, A_crd1, A_pos2, A_crd2, A_vals,
                                ctypes.byref(opts))


def slnr_sddmm_spmm_gemm(B, C, D, K, F, L, W, M, A, opts):
    return lib().slnr_sddmm_spmm_gemm(ctypes.byref(B), C, D, K, F, L, W, M, A, ctypes.byref(opts))


def slnr_mttkrp_gemm(B, C, D, L, E, M, A, opts):
    return lib().slnr_mttkrp_gemm(ctypes.byref(B), C, D, L, E, M, A, ctypes.byref(opts))


def slnr_spmmh_gemm(B, C, D, J, E, L, A, opts):
    return lib().slnr_spmmh_gemm(ctypes.byref(B), C, D, J, E, L, A, ctypes.byref(opts))


def _query(fn_name, *args):
    n = ctypes.c_size_t(0)
    _check(getattr(lib(), fn_name)(*args, ctypes.byref(n)), fn_name)
    return int(n.value)


# ---- torch-facing wrappers ---------------------------------------------------------------

def _torch():
    import torch
    return torch


@dataclass
class DeviceCSR:
    """CSR matrix whose arrays are torch CUDA tensors (int32 pos/crd, fp32 vals)."""
    nrows: int
    ncols: int
    pos: object
    crd: object
    vals: object

    @property
    def nnz(self) -> int:
        return int(self.crd.shape[0])

    @classmethod
    def from_host(cls, B, device="cuda"):
        torch = _torch()
        t = lambda a, dt: torch.as_tensor(a).to(device=device, dtype=dt).contiguous()
        return cls(B.nrows, B.ncols, t(B.pos, torch.int32), t(B.crd, torch.int32), t(B.vals, torch.float32))

    def c_struct(self, vals=None) -> slnr_csr:
        v = self.vals if vals is None else vals
        return slnr_csr(self.nrows, self.ncols, self.nnz, self.pos.data_ptr(), self.crd.data_ptr(), v.data_ptr())


@dataclass
class DeviceCSF3:
    """CSF 3-tensor (levels i -> j -> k) whose arrays are torch CUDA tensors."""
    dims: tuple
    pos1: object
    crd1: object
    pos2: object
    crd2: object
    pos3: object
    crd3: object
    vals: object

    @property
    def nnz(self) -> int:
        return int(self.crd3.shape[0])

    @property
    def nslices(self) -> int:
        return int(self.crd1.shape[0])

    @property
    def nfibers(self) -> int:
        return int(self.crd2.shape[0])

    @classmethod
    def from_host(cls, B, device="cuda"):
        torch = _torch()
        t = lambda a, dt: torch.as_tensor(a).to(device=device, dtype=dt).contiguous()
        i32 = torch.int32
        return cls(tuple(B.dims), t(B.pos1, i32), t(B.crd1, i32), t(B.pos2, i32), t(B.crd2, i32), t(B.pos3, i32),
                   t(B.crd3, i32), t(B.vals, torch.float32))

    def c_struct(self) -> slnr_csf3:
        s = slnr_csf3()
        s.dim[0], s.dim[1], s.dim[2] = self.dims
        s.nnz, s.nslices, s.nfibers = self.nnz, self.nslices, self.nfibers
        s.pos1, s.crd1, s.pos2, s.crd2 = (self.pos1.data_ptr(), self.crd1.data_ptr(), self.pos2.data_ptr(),
                                          self.crd2.data_ptr())
        s.pos3, s.crd3, s.vals = self.pos3.data_ptr(), self.crd3.data_ptr(), self.vals.data_ptr()
        return s


class Workspace:
    """Caller-owned device scratch for the library, grown on demand (one per stream)."""

    def __init__(self, device="cuda"):
        self.device = device
        self.buf = None

    def get(self, nbytes: int):
        torch = _torch()
        nbytes = max(int(nbytes), 256)
        if self.buf is None or self.buf.numel() < nbytes:
            self.buf = torch.empty(nbytes, dtype=torch.uint8, device=self.device)
        return self.buf


_default_ws = {}
_last_ws = [None]

# Bits of the device-side flag word (offset 12 of the workspace header).
DEVICE_FLAGS = {1: "position array malformed", 2: "coordinate out of range", 4: "coordinates not increasing",
                8: "inspector bound exceeded", 16: "device wait timed out"}


def device_flags(workspace=None) -> int:
    """Flag word the kernels of the last call on this workspace set (0 = none); synchronises."""
    buf = workspace.buf if workspace is not None else _last_ws[0]
    if buf is None:
        return 0
    return int(buf[12:16].view(_torch().int32).item())


def _opts(variant, allow_tf32, validate, stream):
    torch = _torch()
    v = {"fused": FUSED, "unfused": UNFUSED}.get(variant, variant)
    s = stream if stream is not None else torch.cuda.current_stream()
    return slnr_opts(int(v), int(bool(allow_tf32)), int(bool(validate)), 0, ctypes.c_void_p(s.cuda_stream), None, 0)


def _attach_ws(opts, nbytes, workspace):
    torch = _torch()
    if workspace is None:
        dev = torch.cuda.current_device()
        workspace = _default_ws.setdefault((dev, opts.stream), Workspace(device=f"cuda:{dev}"))
    buf = workspace.get(nbytes)
    _last_ws[0] = buf
    opts.workspace = buf.data_ptr()
    opts.workspace_bytes = buf.numel()
    return buf


def _dense(x, name):
    torch = _torch()
    if not (x.is_cuda and x.dtype == torch.float32 and x.is_contiguous()):
        raise ValueError(f"{name} must be a contiguous float32 CUDA tensor")
    return x


def spmm_gemm(B: DeviceCSR, C, D, out=None, variant="fused", allow_tf32=True, validate=False, workspace=None,
              stream=None):
    """A(i,l) = sum_{j,k} B(i,j) C(j,k) D(k,l)  (<SpMM,GEMM>, Sec. 6.2)."""
    torch = _torch()
    C, D = _dense(C, "C"), _dense(D, "D")
    K, L = C.shape[1], D.shape[1]
    if out is None:
        out = torch.empty((B.nrows, L), dtype=torch.float32, device=C.device)
    o = _opts(variant, allow_tf32, validate, stream)
    bs = B.c_struct()
    n = _query("slnr_spmm_gemm_workspace", ctypes.byref(bs), K, L, ctypes.byref(o))
    _keep = _attach_ws(o, n, workspace)
    _check(slnr_spmm_gemm(bs, C.data_ptr(), K, D.data_ptr(), L, out.data_ptr(), o), "slnr_spmm_gemm")
    return out


def spmm_gemm_original(B: DeviceCSR, C, D, out=None, stream=None):
    """<SpMM,GEMM> as the perfect loop nest i, j, k, l (the comparator of
    Sec. 6.3's case study; slnr_spmm_gemm_original)."""
    torch = _torch()
    C, D = _dense(C, "C"), _dense(D, "D")
    K, L = C.shape[1], D.shape[1]
    if out is None:
        out = torch.empty((B.nrows, L), dtype=torch.float32, device=C.device)
    bs = B.c_struct()
    s = ctypes.c_void_p((stream or torch.cuda.current_stream()).cuda_stream)
    _check(lib().slnr_spmm_gemm_original(ctypes.byref(bs), C.data_ptr(), K, D.data_ptr(), L, out.data_ptr(), s),
           "slnr_spmm_gemm_original")
    return out


def sddmm_spmm(B: DeviceCSR, C, D, E, out=None, variant="fused", allow_tf32=True, validate=False, workspace=None,
               stream=None):
    """A(i,k) = sum_j B(i,j) (sum_l C(i,l) D(j,l)) E(j,k)  (<SDDMM,SpMM>, Fig. 2; Sec. 6.2)."""
    torch = _torch()
    C, D, E = _dense(C, "C"), _dense(D, "D"), _dense(E, "E")
    L, K = C.shape[1], E.shape[1]
    if out is None:
        out = torch.empty((B.nrows, K), dtype=torch.float32, device=C.device)
    o = _opts(variant, allow_tf32, validate, stream)
    bs = B.c_struct()
    n = _query("slnr_sddmm_spmm_workspace", ctypes.byref(bs), L, K, ctypes.byref(o))
    _keep = _attach_ws(o, n, workspace)
    _check(slnr_sddmm_spmm(bs, C.data_ptr(), D.data_ptr(), L, E.data_ptr(), K, out.data_ptr(), o),
           "slnr_sddmm_spmm")
    return out


def mttkrp(B: DeviceCSF3, C, D, out=None, variant="fused", allow_tf32=True, validate=False, workspace=None,
           stream=None):
    """A(i,l) = sum_{j,k} B(i,j,k) C(j,l) D(k,l)  (MTTKRP, Sec. 6.2)."""
    torch = _torch()
    C, D = _dense(C, "C"), _dense(D, "D")
    L = C.shape[1]
    if out is None:
        out = torch.empty((B.dims[0], L), dtype=torch.float32, device=C.device)
    o = _opts(variant, allow_tf32, validate, stream)
    bs = B.c_struct()
    n = _query("slnr_mttkrp_workspace", ctypes.byref(bs), L, ctypes.byref(o))
    _keep = _attach_ws(o, n, workspace)
    _check(slnr_mttkrp(bs, C.data_ptr(), D.data_ptr(), L, out.data_ptr(), o), "slnr_mttkrp")
    return out


def spttm_ttm(B: DeviceCSF3, C, D, out=None, variant="fused", allow_tf32=True, validate=False, workspace=None,
              stream=None):
    """A(i,j,m) = sum_{k,l} B(i,j,k) C(k,l) D(l,m)  (<SpTTM,SpTTM>, Sec. 6.2).

    Returns (pos1, crd1, pos2, crd2, vals): A's two compressed levels and its
    values (nfibers x M)."""
    torch = _torch()
    C, D = _dense(C, "C"), _dense(D, "D")
    L, M = C.shape[1], D.shape[1]
    dev = C.device
    if out is None:
        i32 = torch.int32
        out = (torch.empty(2, dtype=i32, device=dev), torch.empty(max(B.nslices, 1), dtype=i32, device=dev),
               torch.empty(B.nslices + 1, dtype=i32, device=dev), torch.empty(max(B.nfibers, 1), dtype=i32, device=dev),
               torch.empty((B.nfibers, M), dtype=torch.float32, device=dev))
    o = _opts(variant, allow_tf32, validate, stream)
    bs = B.c_struct()
    n = _query("slnr_spttm_ttm_workspace", ctypes.byref(bs), L, M, ctypes.byref(o))
    _keep = _attach_ws(o, n, workspace)
    p1, c1, p2, c2, v = out
    _check(slnr_spttm_ttm(bs, C.data_ptr(), L, D.data_ptr(), M, p1.data_ptr(), c1.data_ptr(), p2.data_ptr(),
                          c2.data_ptr(), v.data_ptr(), o), "slnr_spttm_ttm")
    return p1, c1[:B.nslices], p2, c2[:B.nfibers], v


def sddmm_spmm_gemm(B: DeviceCSR, C, D, F, W, out=None, variant="fused", allow_tf32=True, validate=False,
                    workspace=None, stream=None):
    """A(i,m) = sum_{j,k,l} B(i,j) C(i,k) D(j,k) F(j,l) W(l,m)  (<SDDMM,SpMM,GEMM>, Sec. 6.2)."""
    torch = _torch()
    C, D, F, W = _dense(C, "C"), _dense(D, "D"), _dense(F, "F"), _dense(W, "W")
    K, L, M = C.shape[1], F.shape[1], W.shape[1]
    if out is None:
        out = torch.empty((B.nrows, M), dtype=torch.float32, device=C.device)
    o = _opts(variant, allow_tf32, validate, stream)
    bs = B.c_struct()
    n = _query("slnr_sddmm_spmm_gemm_workspace", ctypes.byref(bs), K, L, M, ctypes.byref(o))
    _keep = _attach_ws(o, n, workspace)
    _check(slnr_sddmm_spmm_gemm(bs, C.data_ptr(), D.data_ptr(), K, F.data_ptr(), L, W.data_ptr(), M,
                                out.data_ptr(), o), "slnr_sddmm_spmm_gemm")
    return out


def mttkrp_gemm(B: DeviceCSF3, C, D, E, out=None, variant="fused", allow_tf32=True, validate=False, workspace=None,
                stream=None):
    """A(i,m) = sum_{j,k,l} B(i,j,k) C(j,l) D(k,l) E(l,m)  (<MTTKRP,GEMM>, Sec. 6.2)."""
    torch = _torch()
    C, D, E = _dense(C, "C"), _dense(D, "D"), _dense(E, "E")
    L, M = C.shape[1], E.shape[1]
    if out is None:
        out = torch.empty((B.dims[0], M), dtype=torch.float32, device=C.device)
    o = _opts(variant, allow_tf32, validate, stream)
    bs = B.c_struct()
    n = _query("slnr_mttkrp_gemm_workspace", ctypes.byref(bs), L, M, ctypes.byref(o))
    _keep = _attach_ws(o, n, workspace)
    _check(slnr_mttkrp_gemm(bs, C.data_ptr(), D.data_ptr(), L, E.data_ptr(), M, out.data_ptr(), o),
           "slnr_mttkrp_gemm")
    return out


def spmmh_gemm(B: DeviceCSR, C, D, E, out=None, variant="fused", allow_tf32=True, validate=False, workspace=None,
               stream=None):
    """A(i,l) = sum_{k,j} B(i,k) C(k,j) D(k,j) E(j,l)  (<SpMMH,GEMM>, Sec. 6.2)."""
    torch = _torch()
    C, D, E = _dense(C, "C"), _dense(D, "D"), _dense(E, "E")
    J, L = C.shape[1], E.shape[1]
    if out is None:
        out = torch.empty((B.nrows, L), dtype=torch.float32, device=C.device)
    o = _opts(variant, allow_tf32, validate, stream)
    bs = B.c_struct()
    n = _query("slnr_spmmh_gemm_workspace", ctypes.byref(bs), J, L, ctypes.byref(o))
    _keep = _attach_ws(o, n, workspace)
    _check(slnr_spmmh_gemm(bs, C.data_ptr(), D.data_ptr(), J, E.data_ptr(), L, out.data_ptr(), o),
           "slnr_spmmh_gemm")
    return out


def run(op: str, B, dense: dict, **kw):
    """Dispatch by operation name with the dense operands of a workload."""
    if op == "spmm_gemm":
        return spmm_gemm(B, dense["C"], dense["D"], **kw)
    if op == "sddmm_spmm":
        return sddmm_spmm(B, dense["C"], dense["D"], dense["E"], **kw)
    if op == "mttkrp":
        return mttkrp(B, dense["C"], dense["D"], **kw)
    if op == "spttm_ttm":
        return spttm_ttm(B, dense["C"], dense["D"], **kw)
    if op == "sddmm_spmm_gemm":
        return sddmm_spmm_gemm(B, dense["C"], dense["D"], dense["F"], dense["W"], **kw)
    if op == "mttkrp_gemm":
        return mttkrp_gemm(B, dense["C"], dense["D"], dense["E"], **kw)
    if op == "spmmh_gemm":
        return spmmh_gemm(B, dense["C"], dense["D"], dense["E"], **kw)
    raise ValueError(op)
