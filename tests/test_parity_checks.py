"""Host checks of the parity harness's own comparisons (no GPU): the residual-norm
check must pass the oracle against itself and reject a run that stopped early, so a
device kernel that skipped late blocks cannot pass it."""

import numpy as np
import pytest

from oracle import kashin_oracle as ko
from tests import parity


def _resid(x, eps, iters, P):
    d = ko.decompose(x, eps, iters, P=P)
    return np.linalg.norm(d.r, axis=0) / np.linalg.norm(x, axis=0)


@pytest.fixture(scope="module")
def case():
    rng = np.random.default_rng(5)
    N, M = 256, 12
    x = rng.standard_t(4, size=(N, M)) * 0.015
    eps = ko.sign_mask(9, N)
    return x, eps, ko.POperator(N, eps)


def test_residual_check_accepts_equal_runs(case):
    x, eps, P = case
    r = _resid(x, eps, 16, P)
    parity.check_residuals(r, r)
    parity.check_residuals(r * 1.5, r)          # within the factor band
    parity.check_residuals(r * 50, r)           # far below the fp32 floor: only the floor bound


@pytest.mark.parametrize("short", [6, 8])
def test_residual_check_rejects_fewer_blocks(case, short):
    """A run stopped after half the blocks leaves residuals above the fp32 floor."""
    x, eps, P = case
    r16 = _resid(x, eps, 16, P)
    rs = _resid(x, eps, short, P)
    with pytest.raises(AssertionError):
        parity.check_residuals(rs, r16)


def test_residual_check_rejects_drift_where_resolved(case):
    """Above the fp32 floor the norms must agree to RESID_REL, not just the factor band."""
    x, eps, P = case
    r4 = _resid(x, eps, 4, P)
    assert (r4 >= parity.R_RESOLVED).all()
    with pytest.raises(AssertionError):
        parity.check_residuals(r4 * (1 + 10 * parity.RESID_REL), r4)
