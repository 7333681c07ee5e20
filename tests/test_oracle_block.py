"""Pins for the oracle's block on active latents and its step loop (Sec. 3.3)."""
import numpy as np
import pytest
import torch
import torch.nn.functional as Fn

from oracle import block as B
from oracle import cache as C
from oracle import step as ST
from synth import generate as G, small



def _t(a):
    return torch.from_numpy(np.asarray(a, dtype=np.float64))


F64 = dict(dtype=torch.float64)


def test_layer_norm_matches_torch():
    x = G.random_rows(7, 96, seed=1, scale=3.0)
    ref = Fn.layer_norm(_t(x), (96,), eps=1e-6).numpy()
    assert np.allclose(B.layer_norm(x), ref, rtol=1e-12, atol=1e-12)


def test_gelu_matches_torch_tanh_form_and_limits():
    u = np.linspace(-8, 8, 1001)
    ref = Fn.gelu(_t(u), approximate="tanh").numpy()
    assert np.allclose(B.gelu_tanh(u), ref, rtol=1e-13, atol=1e-15)
    assert B.gelu_tanh(np.array([0.0]))[0] == 0.0
    assert abs(B.gelu_tanh(np.array([10.0]))[0] - 10.0) < 1e-12
    # the tanh form stays within 1e-3 of the exact (erf) GELU
    assert np.max(np.abs(B.gelu_tanh(u) - Fn.gelu(_t(u)).numpy())) < 1e-3


@pytest.mark.parametrize("H,d,M,L", [(1, 8, 3, 5), (2, 16, 4, 33), (4, 32, 9, 70)])
def test_mha_matches_torch_sdpa(H, d, M, L):
    g = np.random.default_rng(H * 100 + L)
    Q, K, V = g.standard_normal((M, H * d)), g.standard_normal((L, H * d)), g.standard_normal((L, H * d))
    got = B.mha(Q, K, V, H)
    split = lambda a: _t(a).reshape(a.shape[0], H, d).transpose(0, 1)
    ref = Fn.scaled_dot_product_attention(split(Q), split(K), split(V)).transpose(0, 1).reshape(M, H * d)
    assert np.allclose(got, ref.numpy(), rtol=1e-12, atol=1e-12)


def test_mha_single_key_and_identical_keys():
    g = np.random.default_rng(0)
    Q = g.standard_normal((5, 32))
    V = g.standard_normal((1, 32))
    assert np.allclose(B.mha(Q, g.standard_normal((1, 32)), V, 2), np.repeat(V, 5, 0), atol=1e-14)
    K = np.repeat(g.standard_normal((1, 32)), 6, 0)
    V6 = g.standard_normal((6, 32))
    assert np.allclose(B.mha(Q, K, V6, 2), np.repeat(V6.mean(0, keepdims=True), 5, 0), atol=1e-14)


def test_mha_key_permutation_invariance():
    g = np.random.default_rng(1)
    Q, K, V = g.standard_normal((4, 32)), g.standard_normal((20, 32)), g.standard_normal((20, 32))
    p = g.permutation(20)
    assert np.allclose(B.mha(Q, K, V, 4), B.mha(Q, K[p], V[p], 4), rtol=1e-12, atol=1e-13)


def _torch_block(x, W, cond, H, idx):
    """The same block assembled from torch.nn modules (fp64), for the active rows."""
    D = x.shape[1]
    sa = torch.nn.MultiheadAttention(D, H, bias=True, batch_first=True, **F64)
    ca = torch.nn.MultiheadAttention(D, H, bias=True, batch_first=True, **F64)
    with torch.no_grad():
        sa.in_proj_weight.copy_(torch.cat([_t(W["Wq"]), _t(W["Wk"]), _t(W["Wv"])]))
        sa.in_proj_bias.copy_(torch.cat([_t(W["bq"]), _t(W["bk"]), _t(W["bv"])]))
        sa.out_proj.weight.copy_(_t(W["Wo"]))
        sa.out_proj.bias.copy_(_t(W["bo"]))
        ca.in_proj_weight.copy_(torch.cat([_t(W["Wqc"]), _t(W["Wkc"]), _t(W["Wvc"])]))
        ca.in_proj_bias.copy_(torch.cat([_t(W["bqc"]), _t(W["bkc"]), _t(W["bvc"])]))
        ca.out_proj.weight.copy_(_t(W["Woc"]))
        ca.out_proj.bias.copy_(_t(W["boc"]))
        ln = torch.nn.LayerNorm(D, eps=1e-6, elementwise_affine=False, **F64)
        up = torch.nn.Linear(D, W["W1"].shape[0], **F64)
        down = torch.nn.Linear(W["W1"].shape[0], D, **F64)
        up.weight.copy_(_t(W["W1"]))
        up.bias.copy_(_t(W["b1"]))
        down.weight.copy_(_t(W["W2"]))
        down.bias.copy_(_t(W["b2"]))
        xt = _t(x)[None]
        n1 = ln(xt)
        q = n1[:, torch.as_tensor(idx)]
        h1 = xt[:, torch.as_tensor(idx)] + sa(q, n1, n1, need_weights=False)[0]
        c = _t(cond)[None]
        h2 = h1 + ca(ln(h1), c, c, need_weights=False)[0]
        y = h2 + down(Fn.gelu(up(ln(h2)), approximate="tanh"))
    return y[0].numpy()


def _setup(seed=0):
    w = small(T=3, Hp=2, Wp=4, D=64, H=4, d=16, F=96, Lc=6, n_samples=2400)
    W = G.block_weights(w, 0)
    # larger weights than the workload's 0.02 so that every branch moves the output
    W = {k: (v * 10).astype(np.float32) for k, v in W.items()}
    x = G.random_rows(w.NT, w.D, seed=seed + 10)
    cond = G.random_rows(w.Lc, w.D, seed=seed + 20)
    return w, W, x, cond


def test_block_matches_torch_nn_composition():
    w, W, x, cond = _setup()
    idx = np.array([0, 3, 4, 11, 23], dtype=np.int32)
    got = B.block_active(x, idx, W, cond, w.H)
    ref = _torch_block(x, W, cond, w.H, idx)
    assert np.allclose(got, ref, rtol=1e-10, atol=1e-10)


def test_active_rows_equal_uncached_rows():
    # keys and values come from all latents, so an active row's output does not
    # depend on which other rows are active
    w, W, x, cond = _setup(1)
    full = B.uncached_block(x, W, cond, w.H)
    for idx in ([5], [0, 7, 9, 22], list(range(w.NT))):
        got = B.block_active(x, np.array(idx), W, cond, w.H)
        assert np.allclose(got, full[idx], rtol=1e-12, atol=1e-12)


def test_token_permutation_equivariance():
    w, W, x, cond = _setup(2)
    p = np.random.default_rng(3).permutation(w.NT)
    full = B.uncached_block(x, W, cond, w.H)
    assert np.allclose(B.uncached_block(x[p], W, cond, w.H), full[p], rtol=1e-11, atol=1e-11)


def _cache_state(w, seed):
    q, s = G.random_cache(w.NT, w.D, seed=seed)
    return q, s


def test_ratio_one_is_the_uncached_block():
    w, W, x, cond = _setup(3)
    q, s = _cache_state(w, 4)
    e = G.random_energy(w.T, seed=5)
    r = ST.cached_layer_step(x, q, s, e, W, cond, w.T, w.N, w.H, 1, 1)
    assert list(r.idx) == list(range(w.NT))
    assert np.allclose(r.y, B.uncached_block(x, W, cond, w.H), rtol=1e-12, atol=1e-12)
    qq, ss, _ = C.quantize_rows(C.round_bf16(r.y_act.astype(np.float32)))
    assert np.array_equal(r.q, qq) and np.array_equal(r.s, ss)


def test_ratio_zero_returns_the_reconstructed_cache():
    w, W, x, cond = _setup(4)
    q, s = _cache_state(w, 6)
    e = G.random_energy(w.T, seed=7)
    r = ST.cached_layer_step(x, q, s, e, W, cond, w.T, w.N, w.H, 0, 1)
    assert len(r.idx) == 0
    assert np.array_equal(r.y, C.dequantize_rows(q, s).astype(np.float64))
    assert np.array_equal(r.q, q) and np.array_equal(r.s, s)


def test_partial_step_merges_fresh_and_cached_rows():
    w, W, x, cond = _setup(5)
    q, s = _cache_state(w, 8)
    e = G.random_energy(w.T, seed=9)
    r = ST.cached_layer_step(x, q, s, e, W, cond, w.T, w.N, w.H, 1, 3)
    K = len(r.idx)
    assert K == 8
    full = B.uncached_block(x, W, cond, w.H)
    inactive = np.setdiff1d(np.arange(w.NT), r.idx)
    assert np.allclose(r.y[r.idx], full[r.idx], rtol=1e-12, atol=1e-12)
    assert np.array_equal(r.y[inactive], C.dequantize_rows(q[inactive], s[inactive]))
    assert np.array_equal(r.q[inactive], q[inactive])


def test_step_loop_at_ratio_one_is_the_uncached_stack():
    w, W0, x0, cond0 = _setup(6)
    Ws = [W0, {k: v[::-1].copy() if v.ndim == 1 else v for k, v in W0.items()}]
    conds = [cond0, cond0[::-1].copy()]
    xs = [x0, G.random_rows(w.NT, w.D, seed=99)]
    e = G.random_energy(w.T, seed=1)
    outs = {}

    def rec(t, l, x, q, s, res):
        outs[(t, l)] = res.y_bf16

    ST.generation(xs, Ws, conds, e, w.T, w.N, w.H, 1, 1, record=rec)
    for t in range(2):
        ref = ST.uncached_stack(xs[t], Ws, conds, w.H)
        assert np.allclose(outs[(t, 1)], ref, rtol=2 ** -7, atol=1e-6)
