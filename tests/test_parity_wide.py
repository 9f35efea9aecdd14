"""Inner widths beyond the specialised kernels: CUDA library vs oracle (GPU).

Every entry point takes any inner width that is a multiple of 4 up to 1024.
Powers of two in [4, 256] run on the specialised kernels (K = 256 with
L <= 64 on the tensor cores); other widths run on the run-time-width kernels
with the same schedules.  Each expression is checked element by element at
widths past 256, at widths that are not powers of two, and at mixed pairs,
in both variants and both contraction precisions, on inputs with heavy rows
(split into chunks) and ragged row tiles.  Widths outside the contract (not
a multiple of 4, or above 1024) are rejected before any launch.
"""
import ctypes

import numpy as np
import pytest

import _parity as P
import oracle
import workloads as wl

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def slnr():
    import paper_2205_11622_gb300 as m
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    m.build()
    m.lib()
    return m


@pytest.fixture(scope="module")
def orc():
    return oracle.get()


def check(slnr, orc, w, variant, allow_tf32):
    B, dense = P.to_device(w)
    out = slnr.run(w.op, B, dense, variant=variant, allow_tf32=allow_tf32)
    torch.cuda.synchronize()
    assert slnr.device_flags() == 0, f"device flags {slnr.device_flags():#x}"
    ref, ref_abs = orc.run(w)
    err = P.rel_err(P.values_of(w.op, out).cpu().numpy(), ref, ref_abs)
    tol = P.tolerance(w.op, allow_tf32, variant)
    assert err <= tol, f"{w.name} {w.dims} {variant} tf32={allow_tf32}: err {err:.3e} > {tol:.1e}"


VARIANTS = [("fused", False), ("fused", True), ("unfused", False), ("unfused", True)]


@pytest.mark.gpu
@pytest.mark.parametrize("K,L", [(256, 64), (256, 256), (512, 64), (64, 512), (1024, 16), (256, 32), (12, 100),
                                 (300, 20), (4, 1024), (100, 4), (256, 512), (512, 512)])
@pytest.mark.parametrize("variant,allow_tf32", VARIANTS)
def test_spmm_gemm_wide(slnr, orc, K, L, variant, allow_tf32):
    # 700 rows of R-MAT degree 10: a few rows above 256 nonzeros (chunks), a ragged last tile
    w = wl.spmm_gemm_rmat(0x51A4 + 11 * K + L, 700, 10, K, L)
    check(slnr, orc, w, variant, allow_tf32)


@pytest.mark.gpu
@pytest.mark.parametrize("L,K", [(512, 64), (64, 1024), (100, 12), (20, 300), (1024, 4)])
@pytest.mark.parametrize("variant", ["fused", "unfused"])
def test_sddmm_spmm_wide(slnr, orc, L, K, variant):
    w = wl.sddmm_spmm_rmat(0x51A4 + 5 * L + K, 600, 12, L, K)
    check(slnr, orc, w, variant, False)


@pytest.mark.gpu
@pytest.mark.parametrize("L", [12, 100, 512, 1024])
@pytest.mark.parametrize("variant,allow_tf32", [("fused", False), ("unfused", False)])
def test_mttkrp_wide(slnr, orc, L, variant, allow_tf32):
    w = wl.mttkrp_zipf(0x51A4 + L, (40, 60, 130), 5000, 1.2, L)
    check(slnr, orc, w, variant, allow_tf32)


@pytest.mark.gpu
@pytest.mark.parametrize("L,M", [(512, 64), (64, 512), (100, 36), (12, 1024)])
@pytest.mark.parametrize("variant,allow_tf32", VARIANTS)
def test_spttm_ttm_wide(slnr, orc, L, M, variant, allow_tf32):
    w = wl.spttm_ttm_powerlaw(0x51A4 + L + 3 * M, (60, 70, 900), 8000, 8.0, 900, L, M)
    check(slnr, orc, w, variant, allow_tf32)


@pytest.mark.gpu
@pytest.mark.parametrize("K,L,M", [(12, 100, 20), (512, 64, 64), (64, 512, 1024), (36, 36, 36)])
@pytest.mark.parametrize("variant,allow_tf32", VARIANTS)
def test_sddmm_spmm_gemm_wide(slnr, orc, K, L, M, variant, allow_tf32):
    w = wl.sddmm_spmm_gemm_rmat(0x51A4 + 7 * K + 3 * L + M, 500, 12, K, L, M)
    check(slnr, orc, w, variant, allow_tf32)


@pytest.mark.gpu
@pytest.mark.parametrize("L,M", [(12, 100), (512, 64), (100, 1024)])
@pytest.mark.parametrize("variant,allow_tf32", VARIANTS)
def test_mttkrp_gemm_wide(slnr, orc, L, M, variant, allow_tf32):
    w = wl.mttkrp_gemm_zipf(0x51A4 + 2 * L + M, (40, 60, 130), 5000, 1.2, L, M)
    check(slnr, orc, w, variant, allow_tf32)


@pytest.mark.gpu
@pytest.mark.parametrize("J,L", [(100, 12), (512, 64), (64, 300)])
@pytest.mark.parametrize("variant,allow_tf32", VARIANTS)
def test_spmmh_gemm_wide(slnr, orc, J, L, variant, allow_tf32):
    w = wl.spmmh_gemm_rmat(0x51A4 + J + 5 * L, 600, 10, J, L)
    check(slnr, orc, w, variant, allow_tf32)


@pytest.mark.gpu
def test_heavy_row_wide(slnr, orc):
    # one 3000-nonzero row (12 chunks) among empty rows, widths past 256
    n, ncols = 33, 4000
    cols = np.sort(np.random.default_rng(4).choice(ncols, size=3000, replace=False))
    r = wl.Rng(8)
    pos = np.asarray([0] * 6 + [3000] * (n - 5), np.int32)
    B = wl.CSR(n, ncols, pos, cols.astype(np.int32), wl.uniform(r, 3000, -1, 1))
    for K, L in ((520, 36), (36, 520)):
        dense = {"C": wl.uniform(r, (ncols, K), -1, 1), "D": wl.uniform(r, (K, L), -1, 1)}
        w = wl.Workload("heavy_wide", "spmm_gemm", B, dense, {"K": K, "L": L})
        for variant in ("fused", "unfused"):
            check(slnr, orc, w, variant, False)


def test_widths_outside_the_contract_are_rejected():
    import paper_2205_11622_gb300 as m
    try:
        lib = m.lib()
    except RuntimeError:
        pytest.skip("libslnr.so not built")
    B = m.slnr_csr(10, 10, 0, 0x1000, 0x2000, 0x3000)
    o = m.slnr_opts(0, 0, 0, 0, None, None, 0)
    n = ctypes.c_size_t(0)
    for K, L, want in ((6, 8, 5), (8, 1028, 5), (1024, 1024, 0), (0, 8, 2), (100, 12, 0)):
        st = lib.slnr_spmm_gemm_workspace(ctypes.byref(B), K, L, ctypes.byref(o), ctypes.byref(n))
        assert st == want, (K, L, st, m.last_error())
        if want != 0:  # the perfect-loop-nest comparator checks its widths the same way, before any launch
            st = lib.slnr_spmm_gemm_original(ctypes.byref(B), ctypes.c_void_p(0x1000), K, ctypes.c_void_p(0x2000), L,
                                             ctypes.c_void_p(0x3000), None)
            assert st == want, (K, L, st, m.last_error())
    assert lib.slnr_spmm_gemm_original(ctypes.byref(B), None, 8, ctypes.c_void_p(0x2000), 8,
                                       ctypes.c_void_p(0x3000), None) == 1
