"""Why block outputs are compared with a per-token (normwise) max relative error.

The stated bar for bf16 block outputs against the fp32/fp64 oracle is 2e-2 max
relative and 5e-3 mean relative, without a denominator.  This test runs the
oracle's block twice on the CPU: once in fp64, once as the ideal bf16
tensor-core block of `bf16_model` (every value that a bf16 tensor-core path
must hold in bf16 rounded to bf16: LN outputs, Q/K/V, P, the attention output,
the FFN hidden layer and the output; nothing else).  Even this ideal bf16 path
exceeds 2e-2 under an elementwise reading with a 0.1 rms floor at D = 1024,
while its per-token normwise error max_j|g-o| / max_j|o| and its mean relative
error stay far below the bar.  The GPU tests therefore use the normwise
reading for "max relative", and hold the element-wise figure to a multiple of
this model's element-wise figure on the same rows.
"""
import numpy as np

import oracle
from bf16_model import block_active, elementwise_rel, normwise_rel
from synth import generate as G, small

B = oracle.block


def test_elementwise_floor_reading_is_out_of_reach_for_bf16_operands():
    w = small(T=4, Hp=16, Wp=16, D=1024, H=16, d=64, F=4096, Lc=40, n_samples=16000)
    W = G.block_weights(w, 0)
    audio = G.audio(w)
    cond = G.cond_tokens(w, audio)
    x = G.latents(w).astype(np.float64)
    idx = np.sort(np.random.default_rng(0).choice(w.NT, 256, replace=False))
    ref = B.block_active(x, idx, W, cond, w.H)
    g = block_active(x, idx, W, cond, w.H)
    normwise, mean_rel = normwise_rel(g, ref)
    assert elementwise_rel(g, ref) > 2e-2   # the floored elementwise reading fails for any bf16 path
    assert normwise < 1e-2 and mean_rel < 5e-3


def test_model_rounds_only_where_stated():
    """With no rounding (values already on the bf16 grid are kept) the model's
    pieces reduce to the oracle's: bf is the identity on bf16 values, and the
    attention with P kept exact equals the oracle's."""
    from bf16_model import bf, mha_bf16_p
    v = G.random_rows(4, 16, seed=5)
    assert np.array_equal(bf(v), v.astype(np.float64))
    rng = np.random.default_rng(1)
    Q, K, V = (rng.standard_normal((3, 8)) for _ in range(3))
    # one key: P = 1 exactly, so the bf16 rounding of P changes nothing
    assert np.allclose(mha_bf16_p(Q, K[:1], V[:1], 2), B.mha(Q, K[:1], V[:1], 2), rtol=0, atol=1e-15)
