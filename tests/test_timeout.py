"""Failure detection: a bounded device-side wait that gives up is reported.

The tensor-core kernel's waits (on its mbarriers, its shared counters and its
tile-index ring) give up after slnr_set_wait_limit cycles.  With a limit far
below the time a tile takes to build, the MMA warp's first wait for a full
tile runs out: the kernel sets the timeout bit of the workspace flag word,
drains the MMAs it issued (with the default limit) and frees its tensor
memory, and a call in validate mode returns SLNR_ERR_TIMEOUT.  Nothing here
faults or hangs the GPU: every wait ends, and the context stays usable, which
the correct call after the timeout checks against the oracle.
"""
import ctypes

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


def test_wait_limit_rejects_negative():
    import paper_2205_11622_gb300 as m
    try:
        lib = m.lib()
    except RuntimeError:
        pytest.skip("libslnr.so not built")
    assert lib.slnr_set_wait_limit(ctypes.c_int64(-1)) == 2
    assert lib.slnr_set_wait_limit(ctypes.c_int64(0)) == 0


@pytest.mark.gpu
@pytest.mark.parametrize("op", ["spmm_gemm", "spttm_ttm"])
def test_short_wait_limit_reports_timeout(slnr, op):
    w = wl.spmm_gemm_rmat(0x51A4 + 77, 6000, 16, 64, 64) if op == "spmm_gemm" else \
        wl.spttm_ttm_powerlaw(0x51A4 + 78, (200, 200, 900), 60000, 8.0, 900, 64, 64)
    B, dense = P.to_device(w)
    lib = slnr.lib()
    assert lib.slnr_set_wait_limit(ctypes.c_int64(1000)) == 0
    try:
        with pytest.raises(slnr.SlnrError) as e:
            slnr.run(w.op, B, dense, variant="fused", allow_tf32=True, validate=True)
        assert e.value.status == 7, str(e.value)
        assert slnr.device_flags() & 16
    finally:
        assert lib.slnr_set_wait_limit(ctypes.c_int64(0)) == 0
    # the default limit again: the same call completes and is correct
    out = slnr.run(w.op, B, dense, variant="fused", allow_tf32=True, validate=True)
    torch.cuda.synchronize()
    assert slnr.device_flags() == 0
    ref, ref_abs = oracle.get().run(w)
    err = P.rel_err(P.values_of(w.op, out).cpu().numpy(), ref, ref_abs)
    assert err <= P.TOL_TF32
