"""Helpers for comparing the CUDA library with the oracle.

Error metric: for every output element e,
    err_e = |gpu_e - oracle_e| / A_abs_e
where A_abs is the oracle's magnitude companion (the same loops on absolute
values).  |gpu - exact| <= c * u * A_abs bounds the rounding of any summation
order, so this is the forward error in units of the worst-case magnitude; it
stays meaningful when values cancel to near zero, where a plain relative error
is not.  Where A_abs_e == 0 the GPU value must be exactly 0.  Tolerances are
the ones stated for the target: 1e-4 on fp32 CUDA-core paths, 5e-3 where TF32
tensor cores are used.  Index outputs are compared bit for bit.
"""
from __future__ import annotations

import numpy as np

TOL_FP32 = 1e-4
TOL_TF32 = 5e-3


def rel_err(gpu, ref, ref_abs) -> float:
    gpu = np.asarray(gpu, dtype=np.float64)
    assert gpu.shape == ref.shape, (gpu.shape, ref.shape)
    if not np.all(np.isfinite(gpu)):
        return float("inf")
    diff = np.abs(gpu - ref)
    zero = ref_abs == 0
    if np.any(diff[zero] != 0):
        return float("inf")
    if not np.any(~zero):
        return 0.0
    return float(np.max(diff[~zero] / ref_abs[~zero]))


CSR_OPS = ("spmm_gemm", "sddmm_spmm", "sddmm_spmm_gemm", "spmmh_gemm")


def to_device(w, device="cuda"):
    import torch

    import paper_2205_11622_gb300 as slnr
    if w.op in CSR_OPS:
        B = slnr.DeviceCSR.from_host(w.B, device)
    else:
        B = slnr.DeviceCSF3.from_host(w.B, device)
    dense = {k: torch.from_numpy(np.ascontiguousarray(v)).to(device) for k, v in w.dense.items()}
    return B, dense


def output_rows(w) -> int:
    if w.op in CSR_OPS:
        return w.B.nrows
    if w.op in ("mttkrp", "mttkrp_gemm"):
        return w.B.dims[0]
    return w.B.nfibers


def values_of(op, out):
    return out[4] if op == "spttm_ttm" else out


def uses_tensor_cores(op, variant="fused") -> bool:
    """Whether the call may contract on TF32 tensor cores when allowed: the
    fused and unfused <SpMM,GEMM>, <SpTTM,SpTTM>, <SpMMH,GEMM> and
    <SDDMM,SpMM,GEMM> (fused: where the dot product and the temporary have
    one width), and the dense GEMM of the unfused <MTTKRP,GEMM> (its fused
    consumer runs in fp32)."""
    if op in ("spmm_gemm", "spttm_ttm", "spmmh_gemm", "sddmm_spmm_gemm"):
        return True
    return variant == "unfused" and op == "mttkrp_gemm"


def tolerance(op, allow_tf32, variant="fused") -> float:
    return TOL_TF32 if (allow_tf32 and uses_tensor_cores(op, variant)) else TOL_FP32
