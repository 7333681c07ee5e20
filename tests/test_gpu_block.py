"""GPU parity of the cached layer step (echo_select + echo_block_step) against the oracle.

Every GPU call is fed the oracle's own state (layer input and cache at that
step and layer), so the two sides see identical inputs; nothing the GPU
produced is fed to the oracle.  Bars: selection indices bit-exact, inactive
rows bit-exact (they are the reconstructed cache), inactive cache rows
untouched, active rows within a per-token normwise max rel of 2e-2 and a
mean rel of 5e-3,
and the cache rows written on the GPU are exactly the quantisation of the
bf16 rows it returned.
"""
import numpy as np
import pytest
import torch

import oracle
from synth import STACK4_7800, TINY_256, WAN_BLOCK_32760, generate as G

pytestmark = pytest.mark.gpu
DEV = "cuda"
F32 = np.float32


@pytest.fixture(scope="module")
def ec():
    from paper_2608_02474_gb300 import build
    build.build()
    from paper_2608_02474_gb300 import echocache
    echocache.lib()
    return echocache


def bf(a):
    return torch.from_numpy(np.ascontiguousarray(a, dtype=F32)).to(DEV, torch.bfloat16)


def rel_err(g, o):
    """(max over tokens of max_j|g-o| / max_j|o|, sum|g-o| / sum|o|); the
    normwise reading of "max relative" is justified in test_tolerance_reading.py."""
    nw = np.abs(g - o).max(axis=-1) / np.abs(o).max(axis=-1)
    return float(nw.max()), float(np.abs(g - o).sum() / np.abs(o).sum())


def gpu_layer(ec, blk, w, x, q, s, e, ratio, full=False):
    dims = ec.BlockDims(w.T, w.N, w.D, w.H, w.d, w.F, w.Lc)
    xd = bf(x)
    qd = torch.from_numpy(q.copy()).to(DEV)
    sd = torch.from_numpy(s.copy()).to(DEV)
    if full:
        idx, K = torch.arange(w.NT, dtype=torch.int32, device=DEV), w.NT
    else:
        idx, K, _ = ec.echo_select(xd, qd, sd, torch.from_numpy(e).to(DEV), w.T, w.N, *ratio)
    y = ec.echo_block_step(blk, dims, xd, idx, K, qd, sd)
    torch.cuda.synchronize()
    assert ec.echo_get_device_error() == 0
    return idx.cpu().numpy(), y, qd, sd


def check_layer(ec, w, res, q_in, s_in, g_idx, y, qd, sd, rows=None):
    assert np.array_equal(g_idx, res.idx)
    g = y.float().cpu().numpy()
    act = res.idx if rows is None else rows
    ya = res.y_act if rows is None else res.y_act_rows
    mx, mean = rel_err(g[act], ya)
    assert mx <= 2e-2 and mean <= 5e-3, (mx, mean)
    inactive = np.setdiff1d(np.arange(w.NT), res.idx)
    ref_inactive = oracle.cache.dequantize_rows(q_in[inactive], s_in[inactive])
    assert np.array_equal(g[inactive], ref_inactive)
    gq, gs = qd.cpu().numpy(), sd.cpu().numpy()
    assert np.array_equal(gq[inactive], q_in[inactive]) and np.array_equal(gs[inactive], s_in[inactive])
    # cache rows written by the step == echo_cache_quant of the bf16 rows it
    # returned (echo_cache_quant is itself pinned bit-exact to the oracle)
    if len(res.idx):
        it = torch.from_numpy(res.idx.astype(np.int64)).to(DEV)
        q2 = torch.empty(len(res.idx), w.D, dtype=torch.int8, device=DEV)
        s2 = torch.empty(len(res.idx), dtype=torch.float32, device=DEV)
        ec.echo_cache_quant(y[it].contiguous(), None, q2, s2)
        assert np.array_equal(gq[res.idx], q2.cpu().numpy())
        assert np.array_equal(gs[res.idx], s2.cpu().numpy())
    return mx, mean


def _trajectory(w, steps, layers, profile="speech"):
    audio = G.audio(w, profile)
    _, e = oracle.energy.audio_energy(audio, w.T)
    e32 = e.astype(F32)
    Ws = [G.block_weights(w, l) for l in range(layers)]
    cond = G.cond_tokens(w, audio)
    x0 = G.latents(w)
    xs = [x0] + [G.step_input(w, x0, t) for t in range(1, steps)]
    rec = []
    oracle.step.generation(xs, Ws, [cond] * layers, e32, w.T, w.N, w.H, w.ratio_num, w.ratio_den,
                           record=lambda t, l, x, q, s, r: rec.append((t, l, x, q.copy(), s.copy(), r)))
    return Ws, cond, e32, rec


def test_tiny_every_step(ec):
    w = TINY_256
    Ws, cond, e32, rec = _trajectory(w, w.steps, w.layers)
    blk = ec.DeviceBlock.from_host(Ws[0], cond)
    for t, l, x, q, s, r in rec:
        g_idx, y, qd, sd = gpu_layer(ec, blk, w, x, q, s, e32, (w.ratio_num, w.ratio_den),
                                     full=t == 0)
        check_layer(ec, w, r, q, s, g_idx, y, qd, sd)


def test_stack4_first_steps(ec):
    w = STACK4_7800
    Ws, cond, e32, rec = _trajectory(w, 3, w.layers)
    blks = [ec.DeviceBlock.from_host(W, cond) for W in Ws]
    for t, l, x, q, s, r in rec:
        g_idx, y, qd, sd = gpu_layer(ec, blks[l], w, x, q, s, e32, (w.ratio_num, w.ratio_den),
                                     full=t == 0)
        check_layer(ec, w, r, q, s, g_idx, y, qd, sd)


@pytest.mark.parametrize("profile", ["silence", "tone", "beats"])
def test_tiny_profiles(ec, profile):
    w = TINY_256
    Ws, cond, e32, rec = _trajectory(w, 3, 1, profile)
    blk = ec.DeviceBlock.from_host(Ws[0], cond)
    for t, l, x, q, s, r in rec[1:]:
        g_idx, y, qd, sd = gpu_layer(ec, blk, w, x, q, s, e32, (w.ratio_num, w.ratio_den))
        check_layer(ec, w, r, q, s, g_idx, y, qd, sd)


def test_edge_ratios_and_aliasing(ec):
    w = TINY_256
    W = G.block_weights(w, 0)
    audio = G.audio(w)
    cond = G.cond_tokens(w, audio)
    x = G.latents(w)
    q, s = oracle.cache.quantize_rows(G.step_input(w, x, 2))[:2]
    e = G.random_energy(w.T, seed=1)
    blk = ec.DeviceBlock.from_host(W, cond)
    dims = ec.BlockDims(w.T, w.N, w.D, w.H, w.d, w.F, w.Lc)
    # K = 0: the output is the reconstructed cache, the cache is untouched
    qd, sd = torch.from_numpy(q.copy()).to(DEV), torch.from_numpy(s.copy()).to(DEV)
    y = ec.echo_block_step(blk, dims, bf(x), None, 0, qd, sd)
    assert np.array_equal(y.float().cpu().numpy(), oracle.cache.dequantize_rows(q, s))
    assert np.array_equal(qd.cpu().numpy(), q)
    # K = NT equals the uncached block; y may alias x
    r = oracle.step.cached_layer_step(x, q, s, e, W, cond, w.T, w.N, w.H, 1, 1)
    xd = bf(x)
    qd, sd = torch.from_numpy(q.copy()).to(DEV), torch.from_numpy(s.copy()).to(DEV)
    idx = torch.arange(w.NT, dtype=torch.int32, device=DEV)
    ec.echo_block_step(blk, dims, xd, idx, w.NT, qd, sd, y=xd)
    mx, mean = rel_err(xd.float().cpu().numpy(), oracle.block.uncached_block(x, W, cond, w.H))
    assert mx <= 2e-2 and mean <= 5e-3
    assert ec.echo_get_device_error() == 0


@pytest.mark.slow
@pytest.mark.parametrize("name,layer,step", [("wan_block_32760", 0, 1),
                                             ("wan_stack40_32760", 39, 1),
                                             ("wan_stack40_32760", 19, 10),
                                             ("wan_stack40_32760", 0, 19),
                                             ("wan_sweep_63960", 0, 1)])
def test_wan_block_sampled_rows(ec, name, layer, step):
    """Full-size Wan2.2-S2V-shaped blocks (D 5120, 40 heads) at r = 1/5: the
    32760-token block, layers 0, 19 and 39 of the 40-layer stack (each with its
    own weights) at steps 1, 10 and 19, and the 63960-token sweep shape.  Each
    case is teacher-forced: the layer input is the step-t input and the cache
    holds the quantised step-(t-1) input, as if that had been the previous
    output.  Indices bit-exact, inactive rows bit-exact, 64 sampled active rows
    (32 random, 32 of highest score) against the oracle with keys/values over
    all tokens."""
    from synth import ALL
    w = ALL[name]
    audio = G.audio(w)
    _, e = oracle.energy.audio_energy(audio, w.T)
    e32 = e.astype(F32)
    W = G.block_weights(w, layer)
    cond = G.cond_tokens(w, audio)
    x0 = G.latents(w)
    prev = x0 if step == 1 else G.step_input(w, x0, step - 1)
    x1 = G.step_input(w, x0, step)
    q, s, _ = oracle.cache.quantize_rows(prev)    # cache as if the previous output were prev
    blk = ec.DeviceBlock.from_host(W, cond)
    g_idx, y, qd, sd = gpu_layer(ec, blk, w, x1, q, s, e32, (w.ratio_num, w.ratio_den))

    oidx, osc = oracle.select.select(x1, q, s, e32, w.T, w.N, w.ratio_num, w.ratio_den)
    assert np.array_equal(g_idx, oidx)
    rng = np.random.default_rng(0)
    top = oidx[np.argsort(-osc[oidx], kind="stable")[:32]]
    rows = np.unique(np.concatenate([rng.choice(oidx, 32, replace=False), top]))
    Kv, Vv = oracle.block.self_kv(x1, W)
    Kc, Vc = oracle.block.cross_kv(cond, W)
    ya = oracle.block.active_rows(x1, rows, W, w.H, Kv, Vv, Kc, Vc)

    class R:
        pass
    res = R()
    res.idx, res.y_act_rows = oidx, ya
    check_layer(ec, w, res, q, s, g_idx, y, qd, sd, rows=rows)


def test_pipeline_host_buffers_match_device_steps(ec):
    """CachedStack.run_host (pinned host in/out, copies overlapped with compute)
    returns exactly what the same steps return from device tensors."""
    from paper_2608_02474_gb300.pipeline import CachedStack
    w = TINY_256
    audio = G.audio(w)
    W = G.block_weights(w, 0)
    cond = G.cond_tokens(w, audio)
    x0 = G.latents(w)
    xs = [G.step_input(w, x0, t) for t in (1, 2, 3)]
    blk = ec.DeviceBlock.from_host(W, cond)
    ad = torch.from_numpy(audio).to(DEV)
    outs = []
    for mode in ("device", "host"):
        st = CachedStack(w.T, w.N, w.D, w.H, w.d, w.F, w.Lc, [blk], device=DEV)
        st.set_audio(ad)
        st.step(bf(x0), 1, 1, full=True)
        if mode == "device":
            outs.append([st.step(bf(x), w.ratio_num, w.ratio_den).float().cpu().numpy().copy()
                         for x in xs])
        else:
            hx = [torch.from_numpy(x).to(torch.bfloat16).pin_memory() for x in xs]
            hy = [torch.empty(w.NT, w.D, dtype=torch.bfloat16).pin_memory() for _ in xs]
            st.run_host(hx, hy, w.ratio_num, w.ratio_den)
            torch.cuda.synchronize()
            outs.append([y.float().numpy().copy() for y in hy])
    for a, b in zip(*outs):
        assert np.array_equal(a, b)
    assert ec.echo_get_device_error() == 0
