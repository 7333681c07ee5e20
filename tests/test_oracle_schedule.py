"""Pins for the oracle's step-level adaptive ratio (Sec. 3.3 with Eq. 1)."""
import numpy as np
import pytest

from oracle import schedule as S
from synth import generate as G


def test_delta_of_identical_steps_is_zero():
    h = G.random_rows(50, 64, seed=1)
    assert S.step_delta(h, h) == 0.0


@pytest.mark.parametrize("c", [0.5, 0.9, 1.25, -1.0, 3.0])
def test_delta_of_scaled_output_closed_form(c):
    h = G.random_rows(40, 32, seed=2).astype(np.float64)
    n1 = np.abs(h).sum()
    assert S.step_delta(h, c * h, xi=1e-6) == pytest.approx(abs(1 - c) * n1 / (abs(c) * n1 + 1e-6),
                                                          rel=1e-12)


def test_delta_of_zero_pair_and_from_zero():
    z = np.zeros((4, 8))
    h = G.random_rows(4, 8, seed=3).astype(np.float64)
    assert S.step_delta(z, z) == 0.0
    # from zero to h the change is the whole of h: ||h|| / (||h|| + xi)
    assert S.step_delta(z, h) == pytest.approx(np.abs(h).sum() / (np.abs(h).sum() + 1e-6))


def test_rate_is_clipped_and_monotone():
    assert S.update_rate(0.0) == S.R_MIN
    assert S.update_rate(1e9) == S.R_MAX
    assert S.update_rate(1.0) == pytest.approx(S.R_MIN + S.ALPHA)
    rs = [S.update_rate(d) for d in np.linspace(0, 5, 101)]
    assert all(a <= b for a, b in zip(rs, rs[1:]))


def test_budget_and_normalisation():
    assert S.budget(0.0, 100) == 0 and S.budget(1.0, 100) == 100 and S.budget(0.301, 100) == 31
    assert S.normalised(2.0, 4.0) == 0.5 and S.normalised(1.0, 0.0) == 0.0
    # the first cached step has Delta-hat = 1
    assert S.adaptive_budget(0.3, 0.3, 32760) == int(np.ceil((S.R_MIN + S.ALPHA) * 32760))
    assert S.adaptive_budget(0.0, 0.3, 32760) == int(np.ceil(S.R_MIN * 32760))
