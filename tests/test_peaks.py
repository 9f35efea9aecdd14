"""The peak-measuring kernels behind the roofline's denominators.

slnr_peak_ffma / slnr_peak_tf32 time the library's own FFMA and tcgen05
kind::tf32 kernels; slnr_peak_gather times whole-row gathers from a caller
table.  On the CPU: the gather call's argument checks, which run before any
launch.  On the GPU: every peak is positive and finite, the tensor cores
beat the CUDA cores, and gathers from an L2-resident table beat gathers
from a table far larger than L2.
"""
import ctypes
import math

import pytest

torch = pytest.importorskip("torch")


def test_gather_peak_rejects_bad_arguments():
    import paper_2205_11622_gb300 as m
    try:
        lib = m.lib()
    except RuntimeError:
        pytest.skip("libslnr.so not built")
    v = ctypes.c_double(0.0)
    t = ctypes.c_void_p(0x10000)
    for rows, width, want in ((0, 128, 2), (1 << 31, 128, 2), (100, 3, 2), (100, 256, 2), (100, 48, 2)):
        assert lib.slnr_peak_gather(t, rows, width, None, ctypes.byref(v)) == want, (rows, width)
    assert lib.slnr_peak_gather(ctypes.c_void_p(0x10004), 100, 128, None, ctypes.byref(v)) == 5
    assert lib.slnr_peak_gather(None, 100, 128, None, ctypes.byref(v)) == 1
    assert lib.slnr_peak_gather(t, 100, 128, None, None) == 1


@pytest.mark.gpu
def test_peaks_are_ordered():
    import paper_2205_11622_gb300 as m
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    m.build()
    m.lib()
    p = m.peaks(gather_width=128)
    for k in ("ffma_tflops", "tf32_tflops", "l2_gather_gbs", "hbm_gather_gbs"):
        assert math.isfinite(p[k]) and p[k] > 0, (k, p)
    assert p["tf32_tflops"] > p["ffma_tflops"], p
    assert p["l2_gather_gbs"] > p["hbm_gather_gbs"], p
    q = m.peaks(gather_width=16)
    assert q["l2_gather_gbs"] > 0 and q["hbm_gather_gbs"] > 0, q
