"""Planted mistakes in copies of the oracle must fail the pins (no GPU).

Each case copies oracle/oracle.c, changes one line inside one function (a
dropped factor, a flipped sign, a transposed or wrong index, a lost reset or
accumulation), compiles the copy and runs the pins of tests/_pins.py against
it.  A mutant that passes every pin would mean the pins cannot see that kind
of mistake.  Every mutated index stays inside its array.
"""
import os

import pytest

import _pins
import oracle

FUNCS = ["oracle_spmm_gemm(", "oracle_sddmm_spmm(", "oracle_mttkrp(", "oracle_spttm_ttm(",
         "oracle_spttm_ttm_pattern(", "oracle_sddmm_spmm_gemm(", "oracle_mttkrp_gemm(", "oracle_spmmh_gemm("]

MUTANTS = [
    ("oracle_spmm_gemm(", "t[k] += b * c;", "t[k] += c;"),
    ("oracle_spmm_gemm(", "acc += t[k] * d;", "acc -= t[k] * d;"),
    ("oracle_spmm_gemm(", "D[(int64_t)k * L + l]", "D[(int64_t)l * K + k]"),
    ("oracle_spmm_gemm(", "for (int32_t p = pos[i]; p", "for (int32_t p = pos[i] + 1; p"),
    ("oracle_spmm_gemm(", "C[(int64_t)j * K + k]", "C[(int64_t)(j > 0 ? j - 1 : 0) * K + k]"),
    ("oracle_spmm_gemm(", "ta[k] += fabs(b) * fabs(c);", "ta[k] += b * fabs(c);"),
    ("oracle_sddmm_spmm(", "y += b * c * d;", "y += c * d;"),
    ("oracle_sddmm_spmm(", "C[(int64_t)i * L + l]", "C[(int64_t)(j % nrows) * L + l]"),
    ("oracle_sddmm_spmm(", "a[k] += y * e;", "a[k] += y * e * b;"),
    ("oracle_sddmm_spmm(", "E[(int64_t)j * K + k]", "E[(int64_t)(i % ncols) * K + k]"),
    ("oracle_mttkrp(", "a[l] += t[l] * c;", "a[l] = t[l] * c;"),
    ("oracle_mttkrp(", "C[(int64_t)j * L + l]", "C[(int64_t)(i % d1) * L + l]"),
    ("oracle_mttkrp(", "t[l] += b * d;", "t[l] += d;"),
    ("oracle_mttkrp(", "D[(int64_t)k * L + l]", "D[(int64_t)(j % d2) * L + l]"),
    ("oracle_mttkrp(", "if (crd1[q] != i) continue;", "if (q != i) continue;"),
    ("oracle_spttm_ttm(", "D[(int64_t)l * M + m]", "D[(int64_t)m * L + l]"),
    ("oracle_spttm_ttm(", "t[l] = 0.0;", "(void)0;"),
    ("oracle_spttm_ttm(", "t[l] += b * c;", "t[l] += b * b * c;"),
    ("oracle_spttm_ttm(", "A[s * M + m] = acc;", "A[s * M + m] = acc_abs;"),
    ("oracle_spttm_ttm_pattern(", "A_crd2[nf++] = crd2[f];", "A_crd2[nf++] = crd2[f] + (f == 0);"),
    ("oracle_sddmm_spmm_gemm(", "y += b * c * d;", "y += c * d;"),
    ("oracle_sddmm_spmm_gemm(", "t[l] += y * f;", "t[l] += f;"),
    ("oracle_sddmm_spmm_gemm(", "W[(int64_t)l * M + m]", "W[(int64_t)m * L + l]"),
    ("oracle_sddmm_spmm_gemm(", "C[(int64_t)i * K + k]", "C[(int64_t)(j % nrows) * K + k]"),
    ("oracle_sddmm_spmm_gemm(", "t[l] = 0.0;", "(void)0;"),
    ("oracle_sddmm_spmm_gemm(", "F[(int64_t)j * L + l]", "F[(int64_t)(i % ncols) * L + l]"),
    ("oracle_mttkrp_gemm(", "u[l] += t[l] * c;", "u[l] = t[l] * c;"),
    ("oracle_mttkrp_gemm(", "E[(int64_t)l * M + m]", "E[(int64_t)m * L + l]"),
    ("oracle_mttkrp_gemm(", "t[l] += b * d;", "t[l] += d;"),
    ("oracle_mttkrp_gemm(", "u[l] = 0.0;", "(void)0;"),
    ("oracle_mttkrp_gemm(", "if (crd1[q] != i) continue;", "if (q != i) continue;"),
    ("oracle_mttkrp_gemm(", "C[(int64_t)j * L + l]", "C[(int64_t)(i % d1) * L + l]"),
    ("oracle_spmmh_gemm(", "t[j] += b * c * d;", "t[j] += b * c;"),
    ("oracle_spmmh_gemm(", "t[j] += b * c * d;", "t[j] += b * c * c;"),
    ("oracle_spmmh_gemm(", "E[(int64_t)j * L + l]", "E[(int64_t)l * J + j]"),
    ("oracle_spmmh_gemm(", "acc += t[j] * e;", "acc -= t[j] * e;"),
    ("oracle_spmmh_gemm(", "D[(int64_t)k * J + j]", "D[(int64_t)(k > 0 ? k - 1 : 0) * J + j]"),
]


def mutate(src: str, func: str, old: str, new: str) -> str:
    start = src.index("\n" + ("int64_t " if func == "oracle_spttm_ttm_pattern(" else "int ") + func)
    later = [src.find(f, start + 10) for f in FUNCS]
    later = [x for x in later if x > start]
    end = min(later) if later else len(src)
    body = src[start:end]
    assert body.count(old) >= 1, (func, old)
    return src[:start] + body.replace(old, new, 1) + src[end:]


@pytest.mark.parametrize("idx", range(len(MUTANTS)))
def test_planted_mistake_is_caught(idx, tmp_path):
    func, old, new = MUTANTS[idx]
    src = open(oracle.SOURCE).read()
    mutated = mutate(src, func, old, new)
    assert mutated != src
    c = tmp_path / "mutant.c"
    c.write_text(mutated)
    so = oracle.compile_source(str(c), str(tmp_path / "libmutant.so"))
    fails = _pins.run_all(oracle.Oracle(so), seeds=(1, 2))
    assert fails, f"mutant {idx} ({func} {old!r} -> {new!r}) passed every pin"
