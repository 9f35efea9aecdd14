"""The oracle against facts fixed by the mathematics (no GPU).

See tests/_pins.py for the individual checks: brute-force dense evaluation,
exact integer arithmetic, reductions to scipy.sparse products, closed forms,
the magnitude companion's definition and linearity in every dense operand.
"""
import numpy as np
import pytest

import _pins
import oracle


@pytest.fixture(scope="module")
def orc():
    return oracle.Oracle()


@pytest.mark.parametrize("name", sorted(_pins.ALL_CHECKS))
@pytest.mark.parametrize("seed", [1, 2, 3, 4])
def test_pins(orc, name, seed):
    assert _pins.ALL_CHECKS[name](orc, seed=seed) == []


def test_square_variants(orc):
    assert _pins.check_spmm_gemm(orc, seed=11, square_kl=True) == []
    assert _pins.check_spttm_ttm(orc, seed=11, square_lm=True) == []


def test_zero_nnz(orc):
    pos = np.zeros(5, np.int32)
    e = np.zeros(0, np.int32)
    v = np.zeros(0, np.float32)
    C = np.ones((3, 4), np.float32)
    D = np.ones((4, 2), np.float32)
    A, Aa = orc.spmm_gemm(4, 3, pos, e, v, C, D)
    assert A.shape == (4, 2) and not A.any() and not Aa.any()
    A, _ = orc.sddmm_spmm(4, 4, pos, e, v, np.ones((4, 2), np.float32), np.ones((4, 2), np.float32),
                          np.ones((4, 3), np.float32))
    assert A.shape == (4, 3) and not A.any()
    A, _ = orc.mttkrp((3, 2, 2), e, np.zeros(1, np.int32), e, np.zeros(1, np.int32), e, v,
                      np.ones((2, 4), np.float32), np.ones((2, 4), np.float32))
    assert A.shape == (3, 4) and not A.any()


def test_malformed_input_is_rejected(orc):
    pos = np.array([0, 1], np.int32)
    with pytest.raises(ValueError):
        orc.spmm_gemm(1, 3, pos, np.array([5], np.int32), np.ones(1, np.float32),
                      np.ones((3, 2), np.float32), np.ones((2, 2), np.float32))
    with pytest.raises(ValueError):
        orc.spttm_ttm(3, pos, np.array([-1], np.int32), np.ones(1, np.float32),
                      np.ones((3, 2), np.float32), np.ones((2, 2), np.float32))
