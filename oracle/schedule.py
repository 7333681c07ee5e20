"""Step-level adaptive refresh ratio (Sec. 3.3, "Energy-Guided Step-Latent Cache
Scheduling", with Eq. 1 of Sec. 3.1).

TEST INFRASTRUCTURE ONLY (see the package header).

The paper adjusts the latent update rate of each step from the step-level
change of Eq. 1, Delta_t = ||h_t - h_{t+1}||_1 / (||h_{t+1}||_1 + xi), taken on
the model's intermediate latent output, normalised to Delta-hat_t, as
r_t = clip(r_min + alpha * Delta-hat_t, r_min, r_max), and activates
k_t = ceil(N r_t) latents.  It gives neither the normalisation nor r_min,
r_max, alpha.  Readings:
  * h is the output of the whole cached stack at a step; the change used for
    step t is the most recent one available when step t starts, between the
    outputs of steps t-2 and t-1;
  * Delta-hat = Delta / Delta_ref with Delta_ref the change measured at the
    first cached step (the first Delta available after the full warm-up step),
    so Delta-hat starts at 1; a zero reference leaves Delta-hat = 0;
  * before any change is known (the first cached step) Delta-hat = 1;
  * one global budget K = ceil(r_t * NT) (as for the fixed ratio), computed in
    fp64 and clamped to [0, NT];
  * defaults r_min = 0.1, r_max = 0.5, alpha = 0.2, xi = 1e-6.

Pins: Delta(h, h) = 0; Delta(h, c h) = |1 - c| ||h|| / (|c| ||h|| + xi);
Delta of a zero pair is 0; the clip bounds and monotonicity of r_t; K at the
bounds.
"""
from __future__ import annotations

import math

import numpy as np

R_MIN, R_MAX, ALPHA, XI = 0.1, 0.5, 0.2, 1e-6


def step_sums(h_prev: np.ndarray, h_cur: np.ndarray) -> tuple[float, float]:
    """The two L1 norms of Eq. 1, ||h_prev - h_cur||_1 and ||h_cur||_1, as fp64
    sums of the exact inputs."""
    a = np.asarray(h_prev, dtype=np.float64).ravel()
    b = np.asarray(h_cur, dtype=np.float64).ravel()
    return float(np.abs(a - b).sum()), float(np.abs(b).sum())


def step_delta(h_prev: np.ndarray, h_cur: np.ndarray, xi: float = XI) -> float:
    """Eq. 1 on two consecutive step outputs."""
    num, den = step_sums(h_prev, h_cur)
    return num / (den + xi)


def normalised(delta: float, delta_ref: float) -> float:
    return delta / delta_ref if delta_ref > 0 else 0.0


def update_rate(delta_hat: float, r_min: float = R_MIN, r_max: float = R_MAX,
                alpha: float = ALPHA) -> float:
    return min(max(r_min + alpha * delta_hat, r_min), r_max)


def budget(rate: float, NT: int) -> int:
    return int(min(max(math.ceil(rate * NT), 0), NT))


def adaptive_budget(delta: float, delta_ref: float, NT: int, r_min: float = R_MIN,
                    r_max: float = R_MAX, alpha: float = ALPHA) -> int:
    return budget(update_rate(normalised(delta, delta_ref), r_min, r_max, alpha), NT)


class Schedule:
    """The step loop's state: the Eq. 1 changes seen so far and the budgets
    handed out.  `budget()` gives the next cached step's K from the latest
    change (Delta-hat = 1 before any is known); `observe(h_prev, h_cur)` adds
    the change between two consecutive step outputs."""

    def __init__(self, NT: int, r_min: float = R_MIN, r_max: float = R_MAX, alpha: float = ALPHA,
                 xi: float = XI):
        self.NT, self.r_min, self.r_max, self.alpha, self.xi = NT, r_min, r_max, alpha, xi
        self.deltas: list[float] = []
        self.budgets: list[int] = []

    def budget(self) -> int:
        if self.deltas:
            K = adaptive_budget(self.deltas[-1], self.deltas[0], self.NT, self.r_min, self.r_max,
                                self.alpha)
        else:
            K = budget(update_rate(1.0, self.r_min, self.r_max, self.alpha), self.NT)
        self.budgets.append(K)
        return K

    def observe(self, h_prev: np.ndarray, h_cur: np.ndarray) -> float:
        d = step_delta(h_prev, h_cur, self.xi)
        self.deltas.append(d)
        return d
