"""CUDA library vs oracle, element by element, on seeded inputs (GPU).

Sizes span several row tiles, heavy rows split into chunks, ragged tails,
empty rows / slices, every supported inner width, both variants (fused and
unfused) and both contraction precisions (fp32 and TF32).  Everything goes
through the C ABI (paper_2205_11622_gb300 is a ctypes binding of libslnr).
"""
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


@pytest.fixture(scope="module")
def orc():
    return oracle.get()


def check(slnr, orc, w, variant="fused", allow_tf32=False, tol=None):
    B, dense = P.to_device(w)
    out = slnr.run(w.op, B, dense, variant=variant, allow_tf32=allow_tf32)
    torch.cuda.synchronize()
    assert slnr.device_flags() == 0, f"device flags {slnr.device_flags():#x}"
    ref, ref_abs = orc.run(w)
    got = P.values_of(w.op, out).cpu().numpy()
    err = P.rel_err(got, ref, ref_abs)
    tol = tol if tol is not None else P.tolerance(w.op, allow_tf32, variant)
    assert err <= tol, f"{w.name} {variant} tf32={allow_tf32}: err {err:.3e} > {tol:.1e}"
    if w.op == "spttm_ttm":
        p1, c1, p2, c2 = orc.spttm_ttm_pattern(w.B.crd1, w.B.pos2, w.B.crd2)
        for got_i, want in zip(out[:4], (p1, c1, p2, c2)):
            assert np.array_equal(got_i.cpu().numpy(), want), "output index arrays must be bit-exact"
    return out, err


@pytest.mark.parametrize("idx", range(5))
@pytest.mark.parametrize("variant", ["fused", "unfused"])
@pytest.mark.parametrize("allow_tf32", [False, True])
def test_small_workloads(slnr, orc, idx, variant, allow_tf32):
    check(slnr, orc, wl.small(idx), variant, allow_tf32)


@pytest.mark.parametrize("K,L", [(4, 8), (8, 4), (16, 16), (16, 256), (64, 16), (256, 16), (32, 32), (64, 128),
                                 (128, 64), (128, 128), (128, 256), (256, 256)])
@pytest.mark.parametrize("variant", ["fused", "unfused"])
def test_spmm_gemm_widths(slnr, orc, K, L, variant):
    w = wl.spmm_gemm_rmat(0x51A4 + 7 * K + L, 1537, 12, K, L)
    check(slnr, orc, w, variant, False)
    check(slnr, orc, w, variant, True)


@pytest.mark.parametrize("L,K", [(4, 4), (4, 64), (32, 4), (8, 32), (64, 16), (16, 128), (64, 64), (128, 128), (256, 32)])
@pytest.mark.parametrize("variant", ["fused", "unfused"])
def test_sddmm_spmm_widths(slnr, orc, L, K, variant):
    w = wl.sddmm_spmm_rmat(0x51A4 + 3 * L + K, 1301, 14, L, K)
    check(slnr, orc, w, variant)


@pytest.mark.parametrize("L", [4, 8, 16, 64, 128, 256])
@pytest.mark.parametrize("variant", ["fused", "unfused"])
def test_mttkrp_widths(slnr, orc, L, variant):
    w = wl.mttkrp_zipf(0x51A4 + L, (97, 60, 130), 9000, 1.2, L)
    check(slnr, orc, w, variant)


@pytest.mark.parametrize("L", [4, 32, 256])
@pytest.mark.parametrize("variant", ["fused", "unfused"])
def test_mttkrp_hub_slice(slnr, orc, L, variant):
    # Zipf(1.8) over 40 slices: 3 slices of more than 16 units (512 nonzeros
    # each; the largest has 162, i.e. 3 runs of at most 64 units, the last one
    # ragged) are summed in two levels, the other 37 by a warp each
    w = wl.mttkrp_zipf(0x51A5, (40, 400, 500), 150000, 1.8, L)
    check(slnr, orc, w, variant)


@pytest.mark.parametrize("L,M", [(4, 16), (16, 4), (16, 16), (16, 64), (32, 16), (32, 64), (64, 64), (128, 32),
                                 (128, 256), (256, 128)])
@pytest.mark.parametrize("variant", ["fused", "unfused"])
def test_spttm_ttm_widths(slnr, orc, L, M, variant):
    # 24000 nonzeros: past the size below which the fused call stays on CUDA cores
    w = wl.spttm_ttm_powerlaw(0x51A4 + L + M, (100, 100, 900), 24000, 8.0, 900, L, M)
    check(slnr, orc, w, variant, False)
    check(slnr, orc, w, variant, True)


# ---- edge cases ---------------------------------------------------------------------

def _csr_workload(pos, crd, ncols, K, L, seed=5, op="spmm_gemm"):
    r = wl.Rng(seed)
    nrows = len(pos) - 1
    vals = wl.uniform(r, max(len(crd), 0), -1.0, 1.0)
    B = wl.CSR(nrows, ncols, np.asarray(pos, np.int32), np.asarray(crd, np.int32), vals)
    if op == "spmm_gemm":
        dense = {"C": wl.uniform(r, (ncols, K), -1, 1), "D": wl.uniform(r, (K, L), -1, 1)}
        return wl.Workload("edge", op, B, dense, {"K": K, "L": L})
    dense = {"C": wl.uniform(r, (nrows, L), -1, 1), "D": wl.uniform(r, (ncols, L), -1, 1),
             "E": wl.uniform(r, (ncols, K), -1, 1)}
    return wl.Workload("edge", op, B, dense, {"K": K, "L": L})


@pytest.mark.parametrize("op", ["spmm_gemm", "sddmm_spmm"])
@pytest.mark.parametrize("variant", ["fused", "unfused"])
def test_no_nonzeros(slnr, orc, op, variant):
    w = _csr_workload([0] * 71, [], 50 if op == "spmm_gemm" else 70, 32, 64, op=op)
    out, _ = check(slnr, orc, w, variant)
    assert not torch.any(out != 0)


@pytest.mark.parametrize("op", ["spmm_gemm", "sddmm_spmm"])
@pytest.mark.parametrize("variant", ["fused", "unfused"])
def test_one_heavy_row_among_empty_rows(slnr, orc, op, variant):
    # row 37 holds 5000 nonzeros (20 chunks); every other row is empty; 45 rows (ragged tile)
    n, ncols = 45, 6000
    cols = np.sort(np.random.default_rng(1).choice(ncols, size=5000, replace=False))
    pos = [0] * 38 + [len(cols)] * (n - 37)
    w = _csr_workload(pos, cols.tolist(), ncols, 64, 32, op=op)
    check(slnr, orc, w, variant)


@pytest.mark.parametrize("variant", ["fused", "unfused"])
def test_rows_at_the_split_threshold(slnr, orc, variant):
    # rows with 255, 256, 257, 512, 513 nonzeros straddle the light/heavy boundary and chunk ends
    lens = [255, 256, 257, 512, 513, 1, 0, 3]
    rng = np.random.default_rng(2)
    pos, crd = [0], []
    for l in lens:
        crd += np.sort(rng.choice(700, size=l, replace=False)).tolist()
        pos.append(len(crd))
    check(slnr, orc, _csr_workload(pos, crd, 700, 128, 128), variant)
    check(slnr, orc, _csr_workload(pos, crd, 700, 128, 128), variant, allow_tf32=True)
    w = _csr_workload(pos + [len(crd)] * (700 - len(lens)), crd, 700, 64, 64, op="sddmm_spmm")
    check(slnr, orc, w, variant)


def _csf_workload(op, dims, slices, L, M=None, seed=9):
    """slices: {i: {j: [k...]}} -> CSF workload."""
    r = wl.Rng(seed)
    crd1, pos2, crd2, pos3, crd3 = [], [0], [], [0], []
    for i in sorted(slices):
        crd1.append(i)
        for j in sorted(slices[i]):
            crd2.append(j)
            crd3 += sorted(slices[i][j])
            pos3.append(len(crd3))
        pos2.append(len(crd2))
    a = lambda x: np.asarray(x, np.int32)
    vals = wl.uniform(r, len(crd3), -1, 1)
    B = wl.CSF3(tuple(dims), a([0, len(crd1)]), a(crd1), a(pos2), a(crd2), a(pos3), a(crd3), vals)
    if op == "mttkrp":
        dense = {"C": wl.uniform(r, (dims[1], L), -1, 1), "D": wl.uniform(r, (dims[2], L), -1, 1)}
        return wl.Workload("edge", op, B, dense, {"L": L})
    dense = {"C": wl.uniform(r, (dims[2], L), -1, 1), "D": wl.uniform(r, (L, M), -1, 1)}
    return wl.Workload("edge", op, B, dense, {"L": L, "M": M})


@pytest.mark.parametrize("variant", ["fused", "unfused"])
def test_csf_edges(slnr, orc, variant):
    rng = np.random.default_rng(3)
    # one slice owning everything: a 3000-nonzero fiber (heavy), many short fibers, an empty fiber
    big = {0: sorted(rng.choice(4000, 3000, replace=False).tolist()), 5: [], 7: [1, 2, 3]}
    for j in range(10, 400):
        big[j] = sorted(rng.choice(4000, int(rng.integers(1, 6)), replace=False).tolist())
    slices = {3: big, 11: {}, 12: {2: [5]}}
    for op, L, M in (("mttkrp", 32, None), ("spttm_ttm", 64, 32)):
        w = _csf_workload(op, (20, 400, 4000), slices, L, M)
        out, _ = check(slnr, orc, w, variant)
        if op == "mttkrp":
            ref, _ = orc.run(w)
            assert not ref[0].any() and not out[0].any()  # row without a slice


def test_csf_no_nonzeros(slnr, orc):
    w = _csf_workload("mttkrp", (6, 5, 4), {}, 16)
    out, _ = check(slnr, orc, w)
    assert not torch.any(out != 0)


def test_fused_equals_unfused_and_is_deterministic(slnr, orc):
    for idx in range(1, 5):
        w = wl.small(idx)
        B, dense = P.to_device(w)
        a = P.values_of(w.op, slnr.run(w.op, B, dense, variant="fused", allow_tf32=False)).clone()
        b = P.values_of(w.op, slnr.run(w.op, B, dense, variant="fused", allow_tf32=False)).clone()
        c = P.values_of(w.op, slnr.run(w.op, B, dense, variant="unfused", allow_tf32=False)).clone()
        assert torch.equal(a, b), f"{w.name}: two fused runs differ"
        ref, ref_abs = orc.run(w)
        assert P.rel_err(c.cpu().numpy(), a.cpu().numpy().astype(np.float64), ref_abs) <= 2 * P.TOL_FP32


def test_validate_mode(slnr):
    w = wl.small(2)
    B, dense = P.to_device(w)
    slnr.run(w.op, B, dense, validate=True)  # well-formed: passes
    bad = slnr.DeviceCSR(B.nrows, B.ncols, B.pos, B.crd.clone(), B.vals)
    bad.crd[5] = B.ncols + 3                 # out-of-range coordinate
    with pytest.raises(slnr.SlnrError) as e:
        slnr.run(w.op, bad, dense, validate=True)
    assert e.value.status == 3
    unsorted = slnr.DeviceCSR(B.nrows, B.ncols, B.pos, B.crd.clone(), B.vals)
    r = int(np.argmax(np.diff(w.B.pos)))     # longest row: swap two coordinates
    p = int(w.B.pos[r])
    unsorted.crd[p], unsorted.crd[p + 1] = B.crd[p + 1].item(), B.crd[p].item()
    with pytest.raises(slnr.SlnrError):
        slnr.run(w.op, unsorted, dense, validate=True)
    badpos = slnr.DeviceCSR(B.nrows, B.ncols, B.pos.clone(), B.crd, B.vals)
    badpos.pos[10] = badpos.pos[11] + 1      # non-monotone positions
    with pytest.raises(slnr.SlnrError):
        slnr.run(w.op, badpos, dense, validate=True)
    # CSF: coordinate outside d2
    wc = wl.small(3)
    Bc, dc = P.to_device(wc)
    Bc.crd3 = Bc.crd3.clone()
    Bc.crd3[0] = wc.B.dims[2]
    with pytest.raises(slnr.SlnrError) as e:
        slnr.run(wc.op, Bc, dc, validate=True)
    assert e.value.status == 3


def test_explicit_stream_and_workspace(slnr, orc):
    w = wl.small(4)
    B, dense = P.to_device(w)
    s = torch.cuda.Stream()
    ws = slnr.Workspace()
    with torch.cuda.stream(s):
        out = slnr.run(w.op, B, dense, workspace=ws, stream=s, allow_tf32=False)
    s.synchronize()
    ref, ref_abs = orc.run(w)
    assert P.rel_err(out[4].cpu().numpy(), ref, ref_abs) <= P.TOL_FP32


@pytest.mark.parametrize("K,L", [(32, 64), (64, 64), (128, 128)])
def test_gathered_matrix_larger_than_l2(slnr, orc, K, L):
    # C has 2^20 rows (128-512 MB, more than L2): most gathers miss L2 and
    # reach HBM; 3001 rows of 21 uniform columns give partial last batches
    # in every row
    w = wl.spmm_gemm_uniform(0x51A4 + K + L, 3001, 1 << 20, 21, K, L, name=f"spmm_gemm_wide_{K}")
    check(slnr, orc, w, "fused", True)


@pytest.mark.parametrize("K,L", [(16, 16), (32, 64), (128, 128), (128, 256)])
@pytest.mark.parametrize("nrows", [1, 3, 130])
def test_tiny_inputs(slnr, orc, K, L, nrows):
    # fewer rows than one 128-row tile, exactly one tile plus a ragged second
    # (below 2^14 nonzeros the fused call runs on the CUDA-core kernels)
    w = wl.spmm_gemm_uniform(0x51A4 + 13 * K + L + nrows, nrows, 300, 7, K, L, name=f"tiny_{nrows}")
    check(slnr, orc, w, "fused", True)
    check(slnr, orc, w, "unfused", True)


@pytest.mark.parametrize("K,L", [(128, 256), (256, 16), (256, 64)])
@pytest.mark.parametrize("op", ["spmm_gemm", "spttm_ttm"])
def test_single_buffer_tensor_core_path(slnr, orc, K, L, op):
    # one T buffer (the tile and D^T fill shared memory): waves of short
    # items and single long items make slot ranges that run from one slot
    # tile into the next, over more than 150 tiles; every wait must end
    # (the device flag stays 0) and the result match the oracle
    if op == "spmm_gemm":
        w = wl.spmm_gemm_rmat(0x51A4 + 19 * K + L, 20000, 12, K, L)
    else:
        w = wl.spttm_ttm_powerlaw(0x51A4 + 23 * K + L, (200, 200, 900), 100000, 8.0, 900, K, L)
    check(slnr, orc, w, "fused", True)


@pytest.mark.parametrize("op,size", [("spmm_gemm", "small"), ("spmm_gemm", "large"),
                                     ("sddmm_spmm_gemm", "small"), ("sddmm_spmm_gemm", "large")])
def test_fused_call_routing(slnr, orc, op, size):
    # the fused call takes the tensor-core kernel from 2^14 nonzeros on (TF32
    # allowed, supported widths) and the CUDA-core kernels below; both agree
    # with the oracle
    n, deg = (1024, 10) if size == "small" else (4000, 12)
    w = wl.spmm_gemm_rmat(0x51A4 + 97, n, deg, 64, 64) if op == "spmm_gemm" else \
        wl.sddmm_spmm_gemm_rmat(0x51A4 + 98, n, deg, 64, 64, 64)
    nnz = len(w.B.crd)
    assert (nnz < (1 << 14)) == (size == "small")
    slnr.timing_enable(True)
    try:
        check(slnr, orc, w, "fused", True)
        names = [name for name, _ in slnr.timing_read()]
        launches = slnr.timing_launches()
    finally:
        slnr.timing_enable(False)
    on_tc = any(name.startswith("tc_") for name in names)
    assert on_tc == (size == "large"), names
    # every phase launches at least one kernel; none launches more than two
    assert len(names) <= launches <= 2 * len(names), (names, launches)


@pytest.mark.parametrize("K,L", [(16, 16), (64, 128), (100, 36), (32, 260)])
def test_spmm_gemm_original(slnr, orc, K, L):
    # the perfect loop nest (the case study's comparator): the same A as the
    # oracle; rows of 12 nonzeros keep each output's fp32 chain (12 K terms)
    # within the fp32 tolerance; L = 260 leaves a ragged third column block
    w = wl.spmm_gemm_uniform(0x51A4 + 3 * K + L, 300, 500, 12, K, L, name=f"original_{K}_{L}")
    B, dense = P.to_device(w)
    out = slnr.spmm_gemm_original(B, dense["C"], dense["D"])
    torch.cuda.synchronize()
    ref, ref_abs = orc.run(w)
    assert P.rel_err(out.cpu().numpy(), ref, ref_abs) <= P.TOL_FP32
