"""bench.py's useful-flop counts (the metric's numerator) and byte counts (the
roofline's numerators: referenced rows, every row, gathered rows) against
scalar recounts over the sparse structure, on every small workload and on CSF
tensors with slices that hold no fibers.  The per-unit costs are the fused
schedule's (Sec. 6.2): a dense row product per non-empty row or slice, a vector
update per nonzero and per fiber."""
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


def scalar_bytes(w, referenced_only=True):
    """Bytes an ideal evaluation moves, recounted from the structure: index and
    value arrays once, each dense row read once (only the rows a nonzero, a
    non-empty row or a fiber refers to, with referenced_only), every output
    element once."""
    d, B = w.dims, w.B
    dense = lambda name: w.dense[name] if name in w.dense else None
    if w.op in ("spmm_gemm", "sddmm_spmm", "sddmm_spmm_gemm", "spmmh_gemm"):
        cols = {int(c) for c in B.crd}
        rows = [i for i in range(B.nrows) if B.pos[i + 1] > B.pos[i]]
        total = 4 * (B.nrows + 1) + 8 * len(B.crd)
        if w.op == "spmm_gemm":
            K, L = d["K"], d["L"]
            reads = (len(cols) if referenced_only else B.ncols) * 4 * K + 4 * K * L
            return total + reads + 4 * B.nrows * L
        if w.op == "sddmm_spmm":
            K, L = d["K"], d["L"]
            c_rows = len(rows) if referenced_only else B.nrows
            return total + 4 * L * c_rows + (len(cols) if referenced_only else B.ncols) * 4 * (L + K) + 4 * B.nrows * K
        if w.op == "sddmm_spmm_gemm":
            K, L, M = d["K"], d["L"], d["M"]
            c_rows = len(rows) if referenced_only else B.nrows
            return (total + 4 * K * c_rows + (len(cols) if referenced_only else B.ncols) * 4 * (K + L) + 4 * L * M
                    + 4 * B.nrows * M)
        J, L = d["J"], d["L"]
        return total + (len(cols) if referenced_only else B.ncols) * 8 * J + 4 * J * L + 4 * B.nrows * L
    ns, nf, nnz = len(B.crd1), len(B.crd2), len(B.crd3)
    structure = 8 + 4 * ns + 4 * (ns + 1) + 4 * nf + 4 * (nf + 1) + 8 * nnz
    if w.op == "spttm_ttm":
        L, M = d["L"], d["M"]
        ks = len({int(k) for k in B.crd3}) if referenced_only else B.dims[2]
        out_index = 8 + 4 * ns + 4 * (ns + 1) + 4 * nf
        return structure + 4 * L * ks + 4 * L * M + 4 * nf * M + out_index
    L = d["L"]
    js = len({int(j) for j in B.crd2}) if referenced_only else B.dims[1]
    ks = len({int(k) for k in B.crd3}) if referenced_only else B.dims[2]
    if w.op == "mttkrp_gemm":
        return structure + 4 * L * (js + ks) + 4 * L * d["M"] + 4 * B.dims[0] * d["M"]
    return structure + 4 * L * (js + ks) + 4 * B.dims[0] * L


def scalar_gather_bytes(w):
    """Whole rows the fused producers read: one per nonzero (two for the
    Hadamard and sampled rows), plus one C row per fiber for MTTKRP."""
    d, B = w.dims, w.B
    per = {"spmm_gemm": 4 * d.get("K", 0), "spttm_ttm": 4 * d.get("L", 0), "spmmh_gemm": 8 * d.get("J", 0),
           "sddmm_spmm": 4 * (d.get("L", 0) + d.get("K", 0)), "sddmm_spmm_gemm": 4 * (d.get("K", 0) + d.get("L", 0)),
           "mttkrp": 4 * d.get("L", 0), "mttkrp_gemm": 4 * d.get("L", 0)}[w.op]
    total = 0
    nnz = len(B.crd) if w.op in ("spmm_gemm", "sddmm_spmm", "sddmm_spmm_gemm", "spmmh_gemm") else len(B.crd3)
    for _ in range(nnz):
        total += per
    if w.op in ("mttkrp", "mttkrp_gemm"):
        total += 4 * d["L"] * len(B.crd2)
    return total


@pytest.mark.parametrize("kind,i", CASES)
def test_byte_counts_match_a_recount(kind, i):
    w = wl.small(i) if kind == "small" else wl.next_small(i)
    assert bench.min_bytes(w) == scalar_bytes(w, referenced_only=True)
    assert bench.gather_bytes(w) == scalar_gather_bytes(w)
    assert bench.min_bytes_all_rows(w) == scalar_bytes(w, referenced_only=False)
    assert bench.min_bytes_all_rows(w) >= bench.min_bytes(w)


@pytest.mark.parametrize("width,want", [(4, 4), (12, 8), (32, 32), (100, 64), (128, 128), (512, 128), (1024, 128)])
def test_gather_row_width_is_a_power_of_two_up_to_128(width, want):
    B = wl.CSR(2, 2, np.asarray([0, 1, 1], np.int32), np.asarray([1], np.int32), np.ones(1, np.float32))
    w = wl.Workload("w", "spmm_gemm", B, {}, {"K": width, "L": 8})
    assert bench.gather_row_width(w) == want
