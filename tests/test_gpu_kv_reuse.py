"""K/V kept across steps (echo_block_step_kv, CachedStack(reuse_kv=True)).

Sec. 3.3 takes K and V over the complete latent set at every step.  A token's
K/V row depends on its own layer input only, so recomputing just the rows
whose input changed must give every output bit for bit as recomputing all of
them.  Checked here against echo_block_step on the same inputs, and for whole
stacks against the same stack without reuse.
"""
import numpy as np
import pytest
import torch

import oracle
from synth import STACK4_7800, TINY_256, WAN_STACK40_32760, generate as G

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.fixture(scope="module")
def ec():
    from paper_2608_02474_gb300 import build
    build.build()
    from paper_2608_02474_gb300 import echocache
    echocache.lib()
    return echocache


def bf(a):
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(DEV, torch.bfloat16)


def i32(a):
    return torch.from_numpy(np.asarray(a, dtype=np.int32)).to(DEV)


def kv_of(ec, blk, x):
    """K|V of every row from the exported kernels: LN(x) [Wk; Wv]^T + [bk; bv]."""
    n1 = ec.echo_layernorm(x)
    return ec.echo_linear(n1, blk.tensors["Wkv"], blk.tensors["bkv"])


def test_block_step_kv_equals_block_step(ec):
    w = TINY_256
    W = G.block_weights(w, 0)
    cond = G.cond_tokens(w, G.audio(w))
    blk = ec.DeviceBlock.from_host(W, cond)
    dims = ec.BlockDims(w.T, w.N, w.D, w.H, w.d, w.F, w.Lc)
    rng = np.random.default_rng(0)
    x0 = G.latents(w)
    q, s, _ = oracle.cache.quantize_rows(G.step_input(w, x0, 1))
    kv = torch.empty(w.NT, 2 * w.D, dtype=torch.bfloat16, device=DEV)

    def both(x, idx, K, valid, ra=None, rb=None):
        qa, sa = torch.from_numpy(q.copy()).to(DEV), torch.from_numpy(s.copy()).to(DEV)
        qb, sb = torch.from_numpy(q.copy()).to(DEV), torch.from_numpy(s.copy()).to(DEV)
        ia = i32(idx) if K else None
        ya = ec.echo_block_step(blk, dims, x, ia, K, qa, sa)
        yb = ec.echo_block_step_kv(blk, dims, x, ia, K, kv, valid, qb, sb,
                                   rows_a=None if ra is None else i32(ra), n_a=0 if ra is None else len(ra),
                                   rows_b=None if rb is None else i32(rb), n_b=0 if rb is None else len(rb))
        torch.cuda.synchronize()
        assert ec.echo_get_device_error() == 0
        assert torch.equal(ya, yb) and torch.equal(qa, qb) and torch.equal(sa, sb)
        assert torch.equal(kv, kv_of(ec, blk, x))

    idx = np.sort(rng.choice(w.NT, w.K, replace=False))
    xd0 = bf(x0)
    both(xd0, idx, w.K, False)                         # first call: every row computed
    # change 40 rows of the input; list them over two lists with overlaps
    changed = np.sort(rng.choice(w.NT, 40, replace=False))
    x1 = x0.copy()
    x1[changed] = G.random_rows(40, w.D, seed=7)
    ra, rb = changed[:25], np.concatenate([changed[20:], changed[:3]])
    both(bf(x1), np.sort(rng.choice(w.NT, w.K, replace=False)), w.K, True, ra, rb)
    # K = 0: no block, the kept K/V still follow the input
    x2 = x1.copy()
    x2[changed[:5]] = 0.5
    both(bf(x2), None, 0, True, changed[:5])
    # every row listed, and an empty change with K = NT
    both(bf(x2), np.arange(w.NT), w.NT, True, np.arange(w.NT))
    both(bf(x2), np.arange(w.NT), w.NT, True)


def _stack(ec, w, blocks, reuse):
    from paper_2608_02474_gb300.pipeline import CachedStack
    return CachedStack(w.T, w.N, w.D, w.H, w.d, w.F, w.Lc, blocks, device=DEV, reuse_kv=reuse)


def _compare_stacks(ec, w, steps, layers=None):
    audio = torch.from_numpy(G.audio(w)).to(DEV)
    cond = G.cond_tokens(w, G.audio(w))
    L = layers or w.layers
    blocks = []
    for l in range(L):
        blocks.append(ec.DeviceBlock.from_host(G.block_weights(w, l), cond))
    plain, reuse = _stack(ec, w, blocks, False), _stack(ec, w, blocks, True)
    for st in (plain, reuse):
        st.set_audio(audio)
    for t, x in enumerate(G.step_inputs(w, G.latents(w), steps)):
        xd = bf(x)
        ya = plain.step(xd, w.ratio_num, w.ratio_den, full=t == 0).clone()
        yb = reuse.step(xd, w.ratio_num, w.ratio_den, full=t == 0)
        torch.cuda.synchronize()
        assert ec.echo_get_device_error() == 0
        assert torch.equal(ya, yb), f"step {t}"
    for l in range(L):
        assert torch.equal(plain.cache_q[l], reuse.cache_q[l])
        assert torch.equal(plain.cache_s[l], reuse.cache_s[l])


def test_stack4_reuse_equals_plain(ec):
    """The 7800-token, 4-block stack over all 10 steps: layers 1-3 recompute
    only the rows refreshed at the layer below in this step or the last."""
    _compare_stacks(ec, STACK4_7800, STACK4_7800.steps)


@pytest.mark.slow
def test_stack40_reuse_equals_plain(ec):
    """The 40-layer Wan2.2-S2V-shaped stack, a full step and three cached steps."""
    _compare_stacks(ec, WAN_STACK40_32760, 4)


def test_reuse_with_adaptive_rate_and_random_selection(ec):
    """Reuse under a budget that changes from step to step (the adaptive rate
    of Sec. 3.3) and under the Random selection ablation: still bit for bit."""
    from paper_2608_02474_gb300.pipeline import AdaptiveRate, CachedStack
    w = STACK4_7800
    audio = torch.from_numpy(G.audio(w)).to(DEV)
    cond = G.cond_tokens(w, G.audio(w))
    blocks = [ec.DeviceBlock.from_host(G.block_weights(w, l), cond) for l in range(w.layers)]
    xs = [bf(x) for x in G.step_inputs(w, G.latents(w), 6)]
    for selection in ("energy", "random"):
        outs, budgets = [], []
        for reuse in (False, True):
            st = CachedStack(w.T, w.N, w.D, w.H, w.d, w.F, w.Lc, blocks, device=DEV,
                             selection=selection, reuse_kv=reuse, seed=3)
            st.set_audio(audio)
            rate = AdaptiveRate(w.NT, 0.1, 0.5, 0.2, device=DEV)
            ys = []
            for t, x in enumerate(xs):
                ys.append(st.step_adaptive(x, rate, full=t == 0).clone())
            torch.cuda.synchronize()
            assert ec.echo_get_device_error() == 0
            outs.append(ys)
            budgets.append(list(rate.budgets))
        assert budgets[0] == budgets[1] and len(set(budgets[0])) > 1
        for a, b in zip(*outs):
            assert torch.equal(a, b), selection


def test_resume_with_reuse_matches_the_uninterrupted_run(ec, tmp_path):
    """A stack with K/V kept across steps, its caches saved after three steps
    and loaded into a fresh stack with reuse: the fresh stack recomputes every
    K/V row on its first step and then follows the uninterrupted run bit for
    bit, through steps where only the changed rows are recomputed."""
    w = STACK4_7800
    audio = torch.from_numpy(G.audio(w)).to(DEV)
    cond = G.cond_tokens(w, G.audio(w))
    blocks = [ec.DeviceBlock.from_host(G.block_weights(w, l), cond) for l in range(w.layers)]
    xs = [bf(x) for x in G.step_inputs(w, G.latents(w), 7)]
    a = _stack(ec, w, blocks, True)
    a.set_audio(audio)
    for t in range(3):
        a.step(xs[t], w.ratio_num, w.ratio_den, full=t == 0)
    path = str(tmp_path / "caches.pt")
    a.save_caches(path)
    b = _stack(ec, w, blocks, True)
    b.set_audio(audio)
    b.load_caches(path)
    for t in range(3, 7):
        ya = a.step(xs[t], w.ratio_num, w.ratio_den).clone()
        yb = b.step(xs[t], w.ratio_num, w.ratio_den).clone()
        torch.cuda.synchronize()
        assert ec.echo_get_device_error() == 0
        assert torch.equal(ya, yb), f"step {t}"
