"""The float64 oracle against what the paper and mathematics fix (CPU only)."""
import os
import sys

import pytest

sys.path.insert(0, os.path.dirname(os.path.abspath(__file__)))

import oracle_pins as P


@pytest.mark.parametrize("name", sorted(P.ALL_PINS))
def test_pin(orc, name):
    fn, tol = P.ALL_PINS[name]
    err = fn(orc)
    assert err <= tol, "%s: discrepancy %.3e > %.1e" % (name, err, tol)


@pytest.mark.parametrize("M,S,T", [(4, 7, 7.0), (5, 9, 9.0), (2, 3, 3.0)])
def test_lag_equals_absolute_at_full_resolution(orc, M, S, T):
    """Sec. 3.2 / Alg. 1: the time-rolling form equals the lag form when T = S = 2M-1."""
    assert P.lag_vs_absolute(orc, M, S, T) < 1e-12


@pytest.mark.parametrize("M,S,T", [(4, 4, 16.0), (4, 7, 14.0), (3, 3, 11.0)])
def test_lag_differs_from_absolute_when_blurry(orc, M, S, T):
    """Outside T = S = 2M-1 the two forms are different operators (the permutation argument of
    Sec. 3.2 needs the integer grid), so the oracle must implement one of them: the lag form."""
    assert P.lag_vs_absolute(orc, M, S, T) > 0.1
