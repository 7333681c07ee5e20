"""The seeded input generators: the incremental step inputs equal the direct ones."""
import numpy as np

from synth import generate as G, small


def test_step_inputs_equal_step_input():
    w = small(T=2, Hp=3, Wp=4, D=16)
    x0 = G.latents(w)
    xs = list(G.step_inputs(w, x0, 5))
    assert len(xs) == 5 and np.array_equal(xs[0], x0)
    for t in range(1, 5):
        assert np.array_equal(xs[t], G.step_input(w, x0, t))
