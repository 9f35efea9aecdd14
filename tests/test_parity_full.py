"""Full-size benchmark workloads: CUDA library vs oracle on sampled outputs (GPU).

Each of the five benchmark workloads, and the three further expressions of
Sec. 6.2 (workloads.next_full), is generated at full size and run once
in the launch configuration the benchmark times (fused, TF32 allowed), then
compared with the oracle on sampled output rows: the heaviest rows (split
across chunks), the first and last rows, and a seeded uniform sample.  The
oracle evaluates exactly those rows.
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
    return m


def sample_rows(w, n_uniform=256, n_heavy=24, seed=7):
    rng = np.random.default_rng(seed)
    n = P.output_rows(w)
    if w.op in P.CSR_OPS:
        sizes = np.diff(w.B.pos)
    elif w.op == "spttm_ttm":
        sizes = np.diff(w.B.pos3)
    else:  # mttkrp, mttkrp_gemm: rows are slices' coordinates
        sizes = np.zeros(n, np.int64)
        fib_nnz = np.diff(w.B.pos3)
        slice_nnz = np.add.reduceat(fib_nnz, w.B.pos2[:-1]) if w.B.nfibers else np.zeros(w.B.nslices)
        sizes[w.B.crd1] = slice_nnz
    heavy = np.argsort(sizes)[::-1][:n_heavy]
    rows = np.concatenate([heavy, [0, n - 1], rng.integers(0, n, n_uniform)])
    return np.unique(rows).astype(np.int32)


def _check_full(slnr, w):
    B, dense = P.to_device(w)
    out = slnr.run(w.op, B, dense, variant="fused", allow_tf32=True)
    torch.cuda.synchronize()
    assert slnr.device_flags() == 0, f"device flags {slnr.device_flags():#x}"
    rows = sample_rows(w)
    ref, ref_abs = oracle.get().run(w, rows=rows)
    got = P.values_of(w.op, out)[torch.from_numpy(rows).long().cuda()].cpu().numpy()
    err = P.rel_err(got, ref, ref_abs)
    tol = P.tolerance(w.op, True, "fused")
    assert err <= tol, f"{w.name}: err {err:.3e} > {tol:.1e}"
    if w.op == "spttm_ttm":
        p1, c1, p2, c2 = oracle.get().spttm_ttm_pattern(w.B.crd1, w.B.pos2, w.B.crd2)
        for got_i, want in zip(out[:4], (p1, c1, p2, c2)):
            assert np.array_equal(got_i.cpu().numpy(), want)
    del out
    # unfused variant agrees on the same sample
    out_u = slnr.run(w.op, B, dense, variant="unfused", allow_tf32=True)
    got_u = P.values_of(w.op, out_u)[torch.from_numpy(rows).long().cuda()].cpu().numpy()
    tol_u = P.tolerance(w.op, True, "unfused")
    assert P.rel_err(got_u, ref, ref_abs) <= tol_u


@pytest.mark.parametrize("idx", range(5))
def test_full_size_sampled(slnr, idx):
    _check_full(slnr, wl.full(idx))


@pytest.mark.parametrize("idx", range(3))
def test_next_expressions_full_size_sampled(slnr, idx):
    _check_full(slnr, wl.next_full(idx))
