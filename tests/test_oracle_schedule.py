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


def test_sums_on_a_worked_example():
    # |1-2| + |-2-2| + |3+1| = 9 and |2| + |2| + |-1| = 5
    assert S.step_sums(np.array([1.0, -2.0, 3.0]), np.array([2.0, 2.0, -1.0])) == (9.0, 5.0)
    assert S.step_delta(np.array([1.0, -2.0, 3.0]), np.array([2.0, 2.0, -1.0]), xi=1.0) == 1.5


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


# ---- the adaptive step loop --------------------------------------------------
import oracle  # noqa: E402
from synth import TINY_256  # noqa: E402


def _loop(w, steps, rate=None, ratio=None, same_inputs=False):
    audio = G.audio(w)
    _, e = oracle.energy.audio_energy(audio, w.T)
    W = [G.block_weights(w, 0)]
    cond = [G.cond_tokens(w, audio)]
    x0 = G.latents(w)
    xs = [x0] * steps if same_inputs else [x0] + [G.step_input(w, x0, t) for t in range(1, steps)]
    outs = []
    num, den = ratio or (w.ratio_num, w.ratio_den)
    oracle.step.generation(xs, W, cond, e.astype(np.float32), w.T, w.N, w.H, num, den,
                           record=lambda t, l, x, q, s, r: outs.append(r), rate=rate)
    return outs


def test_pinned_rate_equals_fixed_ratio():
    """r_min = r_max = 1/4: every cached step refreshes ceil(NT / 4) tokens, so
    the adaptive loop is the fixed-ratio loop at 1/4, bit for bit."""
    w = TINY_256
    sch = S.Schedule(w.NT, 0.25, 0.25, 0.7)
    a = _loop(w, 5, rate=sch)
    b = _loop(w, 5, ratio=(1, 4))
    assert sch.budgets == [64] * 4 and len(sch.deltas) == 4
    for ra, rb in zip(a, b):
        assert np.array_equal(ra.idx, rb.idx) and np.array_equal(ra.y_bf16, rb.y_bf16)


def test_first_budgets_use_unit_change_then_follow_delta():
    w = TINY_256
    sch = S.Schedule(w.NT)
    outs = _loop(w, 6, rate=sch)
    k1 = S.budget(S.update_rate(1.0), w.NT)
    # step 1: no change known yet; step 2: Delta-hat = Delta_1 / Delta_1 = 1
    assert sch.budgets[:2] == [k1, k1]
    # step t >= 3 uses the change between the outputs of steps t-2 and t-1,
    # normalised by the first one
    for t in range(3, 6):
        assert sch.budgets[t - 1] == S.adaptive_budget(sch.deltas[t - 2], sch.deltas[0], w.NT)
    assert [len(r.idx) for r in outs[1:]] == sch.budgets
    assert all(d > 0 for d in sch.deltas)


def test_constant_outputs_fall_to_r_min():
    """Identical inputs and a full refresh every step (r_min = r_max = 1) give
    identical outputs: every change is 0.  A second loop with the same inputs
    and alpha = 0 then never leaves r_min."""
    w = TINY_256
    sch = S.Schedule(w.NT, 1.0, 1.0, 0.2)
    _loop(w, 4, rate=sch, same_inputs=True)
    assert sch.deltas == [0.0, 0.0, 0.0]
    sch2 = S.Schedule(w.NT, 0.1, 0.5, 0.0)
    _loop(w, 4, rate=sch2)
    assert sch2.budgets == [26, 26, 26]


def test_large_alpha_saturates_at_r_max_and_full_refresh_matches_uncached():
    w = TINY_256
    sch = S.Schedule(w.NT, 0.1, 1.0, 1e6)
    outs = _loop(w, 4, rate=sch)
    assert sch.budgets == [w.NT] * 3
    # a full refresh at every layer step is the uncached block on that input
    W = G.block_weights(w, 0)
    cond = G.cond_tokens(w, G.audio(w))
    x0 = G.latents(w)
    ref = oracle.step.uncached_stack(G.step_input(w, x0, 3), [W], [cond], w.H)
    assert np.array_equal(outs[3].y_bf16, ref)
