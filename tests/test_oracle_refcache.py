"""Pins for the oracle's cache forms (Sec. 3.4 and the quantisation ablation
of Table 2)."""
import numpy as np
import pytest

from oracle import cache as C
from oracle import refcache as R
from synth import generate as G

F32 = np.float32


def _rows(n, D, seed, smooth=0.0):
    """bf16 rows; with smooth > 0 consecutive rows are correlated (AR(1))."""
    g = np.random.default_rng(seed)
    x = g.standard_normal((n, D)).astype(F32)
    if smooth:
        for i in range(1, n):
            x[i] = smooth * x[i - 1] + np.sqrt(1 - smooth ** 2) * x[i]
    return G.to_bf16_values(x)


def test_similarity_closed_forms():
    x = _rows(6, 64, 1)
    assert np.allclose(R.similarity(x, x), 1.0, atol=1e-6)
    assert np.allclose(R.similarity(x, -x), -1.0, atol=1e-6)
    assert np.allclose(R.similarity(x, 4 * x), 1.0, atol=1e-6)
    e = np.eye(8, dtype=F32)
    assert R.similarity(e[:4], e[4:]).tolist() == [0.0] * 4       # orthogonal: exactly 0
    z = np.zeros((2, 8), dtype=F32)
    assert R.similarity(z, e[:2]).tolist() == [0.0, 0.0]            # zero norm: 0
    # against the fp64 cosine
    y = _rows(6, 64, 2)
    c64 = (x.astype(np.float64) * y).sum(1) / np.linalg.norm(x.astype(np.float64), axis=1) / \
        np.linalg.norm(y.astype(np.float64), axis=1)
    assert np.allclose(R.similarity(x, y), c64, atol=2e-6)


def test_high_tau_makes_every_row_an_exact_reference():
    v = _rows(40, 32, 3, smooth=0.99)
    c = R.RefCache(40, 32, 40, 8, 2.0)
    c.write(np.arange(40), v)
    assert np.array_equal(c.ref, np.arange(40)) and np.all(c.refcount == 1)
    assert np.array_equal(c.reconstruct_bf16(), v) and np.all(c.s == 0)
    assert c.stats() == (40, 40)


def test_unit_segments_make_every_row_a_reference():
    v = _rows(10, 16, 4, smooth=0.99)
    c = R.RefCache(10, 16, 10, 1, -2.0)
    c.write(np.arange(10), v)
    assert np.array_equal(c.ref, np.arange(10))


def test_low_tau_keeps_one_reference_per_segment_within_the_residual_bound():
    D, n, L = 64, 24, 8
    v = _rows(n, D, 5, smooth=0.9)
    c = R.RefCache(n, D, n, L, -2.0)
    c.write(np.arange(n), v)
    assert c.ref.tolist() == [i // L for i in range(n)]
    assert c.refcount.tolist()[:3] == [L] * 3
    xh = c.reconstruct_bf16().astype(np.float64)
    r = v[(np.arange(n) // L) * L].astype(np.float64)
    qs = c.q.astype(np.float64) * c.s[:, None]
    u = 2.0 ** -24
    bound = (c.s[:, None] * (0.5 + 2.0 ** -14) + u * (np.abs(v - r) + np.abs(qs) + np.abs(r + qs))
             + 2.0 ** -8 * np.abs(xh))
    assert np.all(np.abs(v - xh) <= bound)
    # the residual of a smooth row is far smaller than the row: the residual
    # form loses less than plain int8 does on the same rows
    q8, s8, _ = C.quantize_rows(v)
    e_ref = np.abs(v - xh).sum()
    e_int8 = np.abs(v - C.dequantize_rows(q8, s8)).sum()
    assert e_ref < e_int8


def test_empty_pool_is_the_plain_int8_cache():
    NT, D = 30, 32
    a, b = R.RefCache(NT, D, 0, 6, 0.5), R.Int8Cache(NT, D)
    for k, seed in enumerate((6, 7, 8)):
        rows = np.sort(np.random.default_rng(seed).choice(NT, 12, replace=False))
        v = _rows(12, D, seed, smooth=0.95)
        a.write(rows, v)
        b.write(rows, v)
        assert np.array_equal(a.q, b.q) and np.array_equal(a.s, b.s)
        assert np.array_equal(a.reconstruct_bf16(), b.reconstruct_bf16())
        assert np.array_equal(a.reconstruct_f32(), b.reconstruct_f32())
        assert np.all(a.ref == -1)


def test_reference_counts_release_and_reuse():
    NT, D = 48, 16
    c = R.RefCache(NT, D, NT, 8, 0.6)
    g = np.random.default_rng(9)
    for it in range(12):
        rows = np.sort(g.choice(NT, int(g.integers(1, NT + 1)), replace=False))
        c.write(rows, _rows(len(rows), D, 100 + it, smooth=0.8))
        counts = np.bincount(c.ref[c.ref >= 0], minlength=c.R_cap)
        assert np.array_equal(counts, c.refcount)
        live, hw = c.stats()
        assert live == np.count_nonzero(counts) and hw <= NT
    # rewrite every token: all old references are released, the new ones take
    # the lowest slots again
    c.write(np.arange(NT), _rows(NT, D, 7, smooth=0.8))
    live, hw = c.stats()
    assert hw == live


def test_small_pool_falls_back_to_plain_int8_for_late_runs():
    NT, D = 16, 16
    v = _rows(NT, D, 10)                         # uncorrelated: every row a reference
    c = R.RefCache(NT, D, 5, 16, 0.9)
    c.write(np.arange(NT), v)
    assert c.ref.tolist() == list(range(5)) + [-1] * 11
    q8, s8, _ = C.quantize_rows(v[5:])
    assert np.array_equal(c.q[5:], q8) and np.array_equal(c.s[5:], s8)
    assert np.array_equal(c.reconstruct_bf16()[:5], v[:5])


def test_full_cache_keeps_rows():
    c = R.FullCache(8, 16)
    v = _rows(3, 16, 11)
    c.write([1, 4, 6], v)
    assert np.array_equal(c.reconstruct_bf16()[[1, 4, 6]], v)
    assert np.all(c.reconstruct_f32()[[0, 2, 3, 5, 7]] == 0)


def test_layer_step_with_cache_forms():
    """The cache-form layer step: the Int8Cache form is the int8 step bit for
    bit; a FullCache step at r = 0 returns the stored rows; the RefCache form
    with an empty pool is the int8 step."""
    import oracle
    from synth import TINY_256 as w
    audio = G.audio(w)
    _, e = oracle.energy.audio_energy(audio, w.T)
    e32 = e.astype(F32)
    W, cond = G.block_weights(w, 0), G.cond_tokens(w, audio)
    x0 = G.latents(w)
    x1 = G.step_input(w, x0, 1)
    q, s, _ = C.quantize_rows(x0)
    a = oracle.step.cached_layer_step(x1, q, s, e32, W, cond, w.T, w.N, w.H, 1, 4)
    i8 = R.Int8Cache(w.NT, w.D)
    i8.q, i8.s = q.copy(), s.copy()
    b = oracle.step.cached_layer_step_cache(x1, i8, e32, W, cond, w.T, w.N, w.H, 1, 4)
    assert np.array_equal(a.idx, b.idx) and np.array_equal(a.y_bf16, b.y_bf16)
    assert np.array_equal(a.q, b.cache.q) and np.array_equal(a.s, b.cache.s)
    rc = R.RefCache(w.NT, w.D, 0, 8, 0.5)
    rc.q, rc.s = q.copy(), s.copy()
    c = oracle.step.cached_layer_step_cache(x1, rc, e32, W, cond, w.T, w.N, w.H, 1, 4)
    assert np.array_equal(a.idx, c.idx) and np.array_equal(a.y_bf16, c.y_bf16)
    assert np.array_equal(a.q, c.cache.q)
    fc = R.FullCache(w.NT, w.D)
    fc.v = x0.copy()
    d = oracle.step.cached_layer_step_cache(x1, fc, e32, W, cond, w.T, w.N, w.H, 0, 1)
    assert len(d.idx) == 0 and np.array_equal(d.y_bf16, x0)
