"""slnr_sddmm_spmm_noalloc against slnr_sddmm_spmm, through the C ABI (GPU).

The no-allocation entry point is for callers that cannot allocate device
memory (a real-time path that must not enter an allocator, or a host runtime
that owns all device memory): it takes no workspace and uses a fixed 16 MiB
scratch array inside the library.  Calls in a row, on different sizes, must
each agree with the workspace-taking entry point within the fp32 tolerance
of the other parity tests, including a large call followed by a smaller one
and a large one again (the shared array keeps the last call's heavy-row
records, chunks, partial rows and counters) on a graph with rows past the
heavy-row threshold.  Sizes beyond the scratch are rejected with an
explanatory error.  This file is named to run last, and it also passes on
its own in a fresh process.
"""
import ctypes

import numpy as np
import pytest

import _parity as P
import oracle
import workloads as wl

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def slnr():
    import paper_2205_11622_gb300 as m
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    m.build()
    m.lib()
    return m


def _call_both(slnr, w):
    B, dense = P.to_device(w)
    C, D, E = dense["C"], dense["D"], dense["E"]
    L, K = C.shape[1], E.shape[1]
    bs = B.c_struct()
    stream = torch.cuda.current_stream()
    # existing entry point, caller workspace
    A_ref = torch.empty((B.nrows, K), dtype=torch.float32, device="cuda")
    o = slnr.slnr_opts(slnr.FUSED, 0, 0, 0, ctypes.c_void_p(stream.cuda_stream), None, 0)
    need = ctypes.c_size_t(0)
    assert slnr.lib().slnr_sddmm_spmm_workspace(ctypes.byref(bs), L, K, ctypes.byref(o), ctypes.byref(need)) == 0
    ws = torch.empty(max(need.value, 256), dtype=torch.uint8, device="cuda")
    o.workspace, o.workspace_bytes = ws.data_ptr(), ws.numel()
    st = slnr.slnr_sddmm_spmm(bs, C.data_ptr(), D.data_ptr(), L, E.data_ptr(), K, A_ref.data_ptr(), o)
    assert st == 0, slnr.last_error()
    # no-allocation entry point
    A_na = torch.full((B.nrows, K), float("nan"), dtype=torch.float32, device="cuda")
    st = slnr.lib().slnr_sddmm_spmm_noalloc(ctypes.byref(bs), C.data_ptr(), D.data_ptr(), L, E.data_ptr(), K,
                                           A_na.data_ptr(), ctypes.c_void_p(stream.cuda_stream))
    assert st == 0, slnr.last_error()
    torch.cuda.synchronize()
    return A_ref.cpu().numpy(), A_na.cpu().numpy()


def test_noalloc_matches_workspace_entry_point_twice(slnr):
    cases = [wl.small(1), wl.sddmm_spmm_rmat(0x51A4 + 41, 2500, 18, 32, 128)]
    for w in cases:
        ref_ws, got = _call_both(slnr, w)
        _, ref_abs = oracle.get().run(w)
        err = P.rel_err(got, ref_ws.astype(np.float64), ref_abs)
        assert err <= P.TOL_FP32, f"{w.name}: no-alloc differs from slnr_sddmm_spmm by {err:.3e}"


def test_noalloc_large_small_large(slnr):
    # R-MAT hubs: the large graph has rows above the 256-nonzero threshold
    # (split into chunks whose partial rows live in the scratch array)
    large = wl.sddmm_spmm_rmat(0x51A4 + 43, 12000, 24, 64, 64)
    small = wl.sddmm_spmm_rmat(0x51A4 + 44, 900, 6, 16, 32)
    assert int(np.max(np.diff(large.B.pos))) > 256, "the large case must have heavy rows"
    for w in (large, small, large):
        ref_ws, got = _call_both(slnr, w)
        _, ref_abs = oracle.get().run(w)
        err = P.rel_err(got, ref_ws.astype(np.float64), ref_abs)
        assert err <= P.TOL_FP32, f"{w.name}: no-alloc differs from slnr_sddmm_spmm by {err:.3e}"


def test_noalloc_rejects_sizes_beyond_its_scratch(slnr):
    big = slnr.slnr_csr(10_000_000, 10_000_000, 50_000_000, 0x1000, 0x2000, 0x3000)
    st = slnr.lib().slnr_sddmm_spmm_noalloc(ctypes.byref(big), 0x4000, 0x4000, 64, 0x4000, 64, 0x5000, None)
    assert st == 5
    assert "scratch" in slnr.last_error()
