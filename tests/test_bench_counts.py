"""bench.py's useful-flop counts (the metric's numerator) against a scalar
recount over the sparse structure, on every small workload and on CSF tensors
with slices that hold no fibers.  The per-unit costs are the fused schedule's
(Sec. 6.2): a dense row product per non-empty row or slice, a vector update per
nonzero and per fiber."""
import numpy as np
import pytest

import bench
import workloads as wl


def scalar_flops(w):
    d, B = w.dims, w.B
    total = 0
    if w.op in ("spmm_gemm", "sddmm_spmm", "sddmm_spmm_gemm", "spmmh_gemm"):
        for i in range(B.nrows):
            n = int(B.pos[i + 1]) - int(B.pos[i])
            if w.op == "spmm_gemm":
                total += 2 * n * d["K"] + (2 * d["K"] * d["L"] if n else 0)
            elif w.op == "sddmm_spmm":
                total += n * (2 * d["L"] + 1 + 2 * d["K"])
            elif w.op == "sddmm_spmm_gemm":
                total += n * (2 * d["K"] + 1 + 2 * d["L"]) + (2 * d["L"] * d["M"] if n else 0)
            else:
                total += 3 * n * d["J"] + (2 * d["J"] * d["L"] if n else 0)
        return total
    for s in range(len(B.crd1)):
        for f in range(int(B.pos2[s]), int(B.pos2[s + 1])):
            n = int(B.pos3[f + 1]) - int(B.pos3[f])
            if w.op == "spttm_ttm":
                total += 2 * n * d["L"] + 2 * d["L"] * d["M"]
            else:
                total += 2 * n * d["L"] + 2 * d["L"]
        if w.op == "mttkrp_gemm":
            total += 2 * d["L"] * d["M"]
    return total


CASES = [("small", i) for i in range(5)] + [("next", i) for i in range(len(wl.NEXT_OPS))]


@pytest.mark.parametrize("kind,i", CASES)
def test_useful_flops_match_a_scalar_recount(kind, i):
    w = wl.small(i) if kind == "small" else wl.next_small(i)
    assert bench.useful_flops(w) == scalar_flops(w)


def _csf(dims, slices):
    """slices: list of (i, [(j, [k, ...]), ...]); a slice may list no fibers."""
    crd1, pos2, crd2, pos3, crd3 = [], [0], [], [0], []
    for i, fibers in slices:
        crd1.append(i)
        for j, ks in fibers:
            crd2.append(j)
            crd3.extend(ks)
            pos3.append(len(crd3))
        pos2.append(len(crd2))
    a = lambda x: np.asarray(x, np.int32)
    vals = np.ones(len(crd3), np.float32)
    return wl.CSF3(dims, a([0, len(crd1)]), a(crd1), a(pos2), a(crd2), a(pos3), a(crd3), vals)


@pytest.mark.parametrize("op", ["mttkrp", "mttkrp_gemm"])
def test_mttkrp_counts_with_fiberless_slices(op):
    # a slice without fibers in the middle and at the end
    B = _csf((6, 5, 7), [(0, [(1, [0, 3]), (4, [2])]), (2, []), (3, [(0, [1, 2, 6])]), (5, [])])
    dims = {"L": 8, "M": 4} if op == "mttkrp_gemm" else {"L": 8}
    w = wl.Workload("fiberless", op, B, {}, dims)
    assert bench.useful_flops(w) == scalar_flops(w)
    per_row = bench.row_flops(w)
    assert per_row[2] == (2 * 8 * 4 if op == "mttkrp_gemm" else 0)  # a slice without fibers
    assert per_row[1] == 0 and per_row[4] == 0                       # rows without a slice
