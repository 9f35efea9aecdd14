"""The further expressions of Sec. 6.2 -- <SDDMM,SpMM,GEMM>, <MTTKRP,GEMM>
and <SpMMH,GEMM> -- CUDA library vs oracle, element by element (GPU).

As for the four benchmark expressions: several row tiles, heavy rows split
into chunks, ragged tails, empty rows and slices, a range of inner widths
(including ones narrower than the lane layout), both variants and both
contraction precisions, all through the C ABI.
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


def check(slnr, orc, w, variant="fused", allow_tf32=False):
    B, dense = P.to_device(w)
    out = slnr.run(w.op, B, dense, variant=variant, allow_tf32=allow_tf32)
    torch.cuda.synchronize()
    assert slnr.device_flags() == 0, f"device flags {slnr.device_flags():#x}"
    ref, ref_abs = orc.run(w)
    err = P.rel_err(out.cpu().numpy(), ref, ref_abs)
    tol = P.tolerance(w.op, allow_tf32, variant)
    assert err <= tol, f"{w.name} {variant} tf32={allow_tf32}: err {err:.3e} > {tol:.1e}"
    return out


@pytest.mark.parametrize("idx", range(3))
@pytest.mark.parametrize("variant", ["fused", "unfused"])
@pytest.mark.parametrize("allow_tf32", [False, True])
def test_small_workloads(slnr, orc, idx, variant, allow_tf32):
    check(slnr, orc, wl.next_small(idx), variant, allow_tf32)


@pytest.mark.parametrize("K,L,M", [(4, 4, 4), (4, 64, 16), (64, 4, 8), (16, 128, 64), (64, 64, 64),
                                   (128, 32, 256), (256, 256, 32)])
@pytest.mark.parametrize("variant", ["fused", "unfused"])
def test_sddmm_spmm_gemm_widths(slnr, orc, K, L, M, variant):
    w = wl.sddmm_spmm_gemm_rmat(0x51A4 + 5 * K + 3 * L + M, 1301, 14, K, L, M)
    check(slnr, orc, w, variant, False)
    check(slnr, orc, w, variant, True)


@pytest.mark.parametrize("L,M", [(4, 8), (8, 4), (32, 64), (64, 32), (128, 128), (256, 16)])
@pytest.mark.parametrize("variant", ["fused", "unfused"])
def test_mttkrp_gemm_widths(slnr, orc, L, M, variant):
    w = wl.mttkrp_gemm_zipf(0x51A4 + 2 * L + M, (97, 60, 130), 9000, 1.2, L, M)
    check(slnr, orc, w, variant, False)
    check(slnr, orc, w, variant, True)


@pytest.mark.parametrize("L,M", [(4, 8), (32, 64), (256, 16)])
@pytest.mark.parametrize("variant", ["fused", "unfused"])
def test_mttkrp_gemm_hub_slice(slnr, orc, L, M, variant):
    # 3 slices of more than 16 units (two-level sums, the largest in 3 runs of
    # at most 64 units), 37 small ones (a warp each)
    w = wl.mttkrp_gemm_zipf(0x51A5, (40, 400, 500), 150000, 1.8, L, M)
    check(slnr, orc, w, variant, False)
    check(slnr, orc, w, variant, True)


@pytest.mark.parametrize("J,L", [(4, 8), (16, 256), (32, 32), (64, 128), (128, 64), (128, 128), (256, 64)])
@pytest.mark.parametrize("variant", ["fused", "unfused"])
def test_spmmh_gemm_widths(slnr, orc, J, L, variant):
    w = wl.spmmh_gemm_rmat(0x51A4 + 11 * J + L, 1537, 12, J, L)
    check(slnr, orc, w, variant, False)
    check(slnr, orc, w, variant, True)


# ---- edge cases ---------------------------------------------------------------------

def _csr(op, pos, crd, ncols, seed=5):
    r = wl.Rng(seed)
    nrows = len(pos) - 1
    vals = wl.uniform(r, len(crd), -1.0, 1.0)
    B = wl.CSR(nrows, ncols, np.asarray(pos, np.int32), np.asarray(crd, np.int32), vals)
    if op == "sddmm_spmm_gemm":
        dense = {"C": wl.uniform(r, (nrows, 32), -1, 1), "D": wl.uniform(r, (ncols, 32), -1, 1),
                 "F": wl.uniform(r, (ncols, 64), -1, 1), "W": wl.uniform(r, (64, 16), -1, 1)}
        return wl.Workload("edge", op, B, dense, {"K": 32, "L": 64, "M": 16})
    dense = {"C": wl.uniform(r, (ncols, 128), -1, 1), "D": wl.uniform(r, (ncols, 128), -1, 1),
             "E": wl.uniform(r, (128, 64), -1, 1)}
    return wl.Workload("edge", op, B, dense, {"J": 128, "L": 64})


@pytest.mark.parametrize("op", ["sddmm_spmm_gemm", "spmmh_gemm"])
@pytest.mark.parametrize("variant", ["fused", "unfused"])
def test_no_nonzeros(slnr, orc, op, variant):
    out = check(slnr, orc, _csr(op, [0] * 71, [], 70), variant, True)
    assert not torch.any(out != 0)


@pytest.mark.parametrize("op", ["sddmm_spmm_gemm", "spmmh_gemm"])
@pytest.mark.parametrize("variant", ["fused", "unfused"])
def test_rows_at_the_split_thresholds(slnr, orc, op, variant):
    # 127/128/129 straddle the tensor-core segment length, 255/256/257 the
    # light/heavy boundary of the row kernels, 5000 is a long heavy row; a
    # ragged number of rows (not a multiple of any tile)
    lens = [127, 128, 129, 255, 256, 257, 5000, 1, 0, 3] + [0] * 35
    rng = np.random.default_rng(4)
    pos, crd = [0], []
    for l in lens:
        crd += np.sort(rng.choice(6000, size=l, replace=False)).tolist()
        pos.append(len(crd))
    w = _csr(op, pos, crd, 6000)
    check(slnr, orc, w, variant, False)
    check(slnr, orc, w, variant, True)


@pytest.mark.parametrize("variant", ["fused", "unfused"])
def test_mttkrp_gemm_csf_edges(slnr, orc, variant):
    # a hub slice with a 3000-nonzero fiber and many short fibers, a slice
    # with no fiber, rows of A with no slice at all
    rng = np.random.default_rng(3)
    big = {0: sorted(rng.choice(4000, 3000, replace=False).tolist()), 5: [], 7: [1, 2, 3]}
    for j in range(10, 400):
        big[j] = sorted(rng.choice(4000, int(rng.integers(1, 6)), replace=False).tolist())
    slices = {3: big, 11: {}, 12: {2: [5]}}
    r = wl.Rng(9)
    crd1, pos2, crd2, pos3, crd3 = [], [0], [], [0], []
    for i in sorted(slices):
        crd1.append(i)
        for j in sorted(slices[i]):
            crd2.append(j)
            crd3 += sorted(slices[i][j])
            pos3.append(len(crd3))
        pos2.append(len(crd2))
    a = lambda x: np.asarray(x, np.int32)
    dims = (20, 400, 4000)
    B = wl.CSF3(dims, a([0, len(crd1)]), a(crd1), a(pos2), a(crd2), a(pos3), a(crd3),
                wl.uniform(r, len(crd3), -1, 1))
    dense = {"C": wl.uniform(r, (dims[1], 32), -1, 1), "D": wl.uniform(r, (dims[2], 32), -1, 1),
             "E": wl.uniform(r, (32, 64), -1, 1)}
    w = wl.Workload("edge", "mttkrp_gemm", B, dense, {"L": 32, "M": 64})
    out = check(slnr, orc, w, variant, True)
    assert not out[0].any() and not out[11].any()   # no slice / a slice without fibers


def test_fused_is_deterministic_and_agrees_with_unfused(slnr, orc):
    for idx in range(3):
        w = wl.next_small(idx)
        B, dense = P.to_device(w)
        a = slnr.run(w.op, B, dense, variant="fused", allow_tf32=False).clone()
        b = slnr.run(w.op, B, dense, variant="fused", allow_tf32=False).clone()
        c = slnr.run(w.op, B, dense, variant="unfused", allow_tf32=False).clone()
        assert torch.equal(a, b), f"{w.name}: two fused runs differ"
        _, ref_abs = orc.run(w)
        assert P.rel_err(c.cpu().numpy(), a.cpu().numpy().astype(np.float64), ref_abs) <= 2 * P.TOL_FP32


def test_spmmh_gemm_gathered_matrices_larger_than_l2(slnr, orc):
    # C and D have 2^20 rows of 128 floats (1 GB, far more than L2): most of
    # the Hadamard producers' gathers reach HBM
    r = wl.Rng(0x51A4 + 77)
    n, ncols, J, L = 2001, 1 << 20, 128, 64
    pos, crd = wl.uniform_csr_structure(r, n, ncols, 19)
    vals = wl.uniform(r, crd.shape[0], -1.0, 1.0)
    dense = {"C": wl.normal(r, (ncols, J)), "D": wl.normal(r, (ncols, J)), "E": wl.normal(r, (J, L))}
    w = wl.Workload("spmmh_gemm_wide", "spmmh_gemm", wl.CSR(n, ncols, pos, crd, vals), dense, {"J": J, "L": L})
    check(slnr, orc, w, "fused", True)
