"""The C ABI library loads, exports every declared symbol, and its host-side
argument checks behave as documented in include/slnr.h (no GPU needed: no
call here reaches a CUDA API)."""
import ctypes
import os
import re

import pytest

import paper_2205_11622_gb300 as slnr

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "slnr.h")


@pytest.fixture(scope="module")
def lib():
    slnr.build()
    return slnr.lib()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(slnr_[a-z0-9_]+)\s*\(", text)))


def test_header_declares_the_abi():
    names = declared_functions()
    for must in ["slnr_spmm_gemm", "slnr_sddmm_spmm", "slnr_mttkrp", "slnr_spttm_ttm", "slnr_status_string",
                 "slnr_last_error", "slnr_version", "slnr_spmm_gemm_workspace"]:
        assert must in names


def test_every_declared_symbol_is_exported(lib):
    for name in declared_functions():
        assert hasattr(lib, name), f"{name} declared in slnr.h but not exported"
        assert name in slnr.SIGNATURES, f"{name} has no binding signature"


def test_status_strings(lib):
    for code, name in slnr.STATUS.items():
        assert lib.slnr_status_string(code).decode() == name
    assert lib.slnr_version().decode().startswith("slnr")


def _opts(**kw):
    o = slnr.slnr_opts(0, 0, 0, 0, None, None, 0)
    for k, v in kw.items():
        setattr(o, k, v)
    return o


def _csr(nrows=8, ncols=8, nnz=16):
    return slnr.slnr_csr(nrows, ncols, nnz, 0x1000, 0x2000, 0x3000)


def test_workspace_query_and_argument_errors(lib):
    n = ctypes.c_size_t(0)
    B = _csr(1000, 1000, 100_000)
    o = _opts()
    assert lib.slnr_spmm_gemm_workspace(ctypes.byref(B), 32, 64, ctypes.byref(o), ctypes.byref(n)) == 0
    fused = n.value
    assert fused > 0 and fused % 256 == 0
    ou = _opts(variant=1)
    assert lib.slnr_spmm_gemm_workspace(ctypes.byref(B), 32, 64, ctypes.byref(ou), ctypes.byref(n)) == 0
    assert n.value >= fused + 1000 * 32 * 4          # the materialised T
    # inner dimensions: any multiple of 4 in [4, 1024]; others are unsupported
    assert lib.slnr_spmm_gemm_workspace(ctypes.byref(B), 48, 64, ctypes.byref(o), ctypes.byref(n)) == 0
    assert lib.slnr_spmm_gemm_workspace(ctypes.byref(B), 32, 512, ctypes.byref(o), ctypes.byref(n)) == 0
    assert lib.slnr_spmm_gemm_workspace(ctypes.byref(B), 50, 64, ctypes.byref(o), ctypes.byref(n)) == 5
    assert "multiple of 4" in slnr.last_error()
    assert lib.slnr_spmm_gemm_workspace(ctypes.byref(B), 32, 1028, ctypes.byref(o), ctypes.byref(n)) == 5
    assert lib.slnr_spmm_gemm_workspace(ctypes.byref(B), 0, 64, ctypes.byref(o), ctypes.byref(n)) == 2
    # bad options
    assert lib.slnr_spmm_gemm_workspace(ctypes.byref(B), 32, 64, None, ctypes.byref(n)) == 1
    bad = _opts(variant=7)
    assert lib.slnr_spmm_gemm_workspace(ctypes.byref(B), 32, 64, ctypes.byref(bad), ctypes.byref(n)) == 5
    # negative sizes
    Bn = _csr(-1, 8, 0)
    assert lib.slnr_spmm_gemm_workspace(ctypes.byref(Bn), 32, 64, ctypes.byref(o), ctypes.byref(n)) == 2


def test_compute_calls_reject_bad_arguments_before_any_launch(lib):
    B = _csr(64, 64, 100)
    o = _opts(workspace=0x100000, workspace_bytes=1 << 30)
    # NULL dense operand
    assert lib.slnr_spmm_gemm(ctypes.byref(B), None, 32, 0x4000, 32, 0x5000, ctypes.byref(o)) == 1
    # misaligned dense operand
    assert lib.slnr_spmm_gemm(ctypes.byref(B), 0x4004, 32, 0x4000, 32, 0x5000, ctypes.byref(o)) == 5
    # workspace too small / missing / misaligned
    small = _opts(workspace=0x100000, workspace_bytes=16)
    assert lib.slnr_spmm_gemm(ctypes.byref(B), 0x4000, 32, 0x4000, 32, 0x5000, ctypes.byref(small)) == 4
    none = _opts()
    assert lib.slnr_sddmm_spmm(ctypes.byref(B), 0x4000, 0x4000, 32, 0x4000, 32, 0x5000, ctypes.byref(none)) == 4
    mis = _opts(workspace=0x100010, workspace_bytes=1 << 30)
    assert lib.slnr_spmm_gemm(ctypes.byref(B), 0x4000, 32, 0x4000, 32, 0x5000, ctypes.byref(mis)) == 4
    # nnz > 0 with NULL coordinates
    Bnull = slnr.slnr_csr(64, 64, 100, 0x1000, None, None)
    assert lib.slnr_spmm_gemm(ctypes.byref(Bnull), 0x4000, 32, 0x4000, 32, 0x5000, ctypes.byref(o)) == 1


def test_csf_checks(lib):
    n = ctypes.c_size_t(0)
    o = _opts()
    B = slnr.slnr_csf3()
    B.dim[0], B.dim[1], B.dim[2] = 100, 100, 100
    B.nnz, B.nslices, B.nfibers = 5000, 100, 2000
    assert lib.slnr_mttkrp_workspace(ctypes.byref(B), 32, ctypes.byref(o), ctypes.byref(n)) == 0
    assert n.value > 0
    assert lib.slnr_spttm_ttm_workspace(ctypes.byref(B), 64, 64, ctypes.byref(o), ctypes.byref(n)) == 0
    B.nslices = 101  # more slices than d0
    assert lib.slnr_mttkrp_workspace(ctypes.byref(B), 32, ctypes.byref(o), ctypes.byref(n)) == 2


def test_missing_library_fails_loudly(monkeypatch, tmp_path):
    monkeypatch.setattr(slnr, "_lib", None)
    monkeypatch.setattr(slnr, "LIBRARY", str(tmp_path / "nope.so"))
    with pytest.raises(RuntimeError, match="not built"):
        slnr.lib()
