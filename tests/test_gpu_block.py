"""GPU parity of the cached layer step (echo_select + echo_block_step) against the oracle.

The GPU and the oracle always see identical inputs.  In the oracle-trajectory
tests every GPU call is fed the oracle's own state (layer input and cache at
that step and layer).  In the 40-layer test the GPU runs its own trajectory
through CachedStack, and at sampled (step, layer) pairs the oracle is fed the
GPU's layer input, cache and segment energy (teacher forcing, so that bf16
differences never change a later selection).

Bars: selection indices bit-exact, inactive rows bit-exact (they are the
reconstructed cache), inactive cache rows untouched, the cache rows written on
the GPU exactly the quantisation of the bf16 rows it returned; active rows
within a per-token normwise max rel of 2e-2 and a mean rel of 5e-3, and their
element-wise relative error (|g - o| / max(|o|, 0.1 rms)) at most EL_FACTOR
times that of the ideal bf16 tensor-core block (bf16_model) on the same rows.
"""
import numpy as np
import pytest
import torch

import oracle
from bf16_model import elementwise_rel, normwise_rel
import bf16_model as M
from synth import STACK4_7800, TINY_256, WAN_BLOCK_32760, WAN_STACK40_32760, WAN_SWEEP_63960
from synth import generate as G

pytestmark = pytest.mark.gpu
DEV = "cuda"
F32 = np.float32
# The GPU's element-wise error may exceed the ideal bf16 block's by this factor:
# beyond the model's roundings it accumulates in fp32 in tile order, takes exp2
# from the hardware's approximation, and rounds P to bf16 against a running
# maximum taken from the first key block rather than the row's true maximum.
# Measured on GB300 the ratio stayed within 0.86-1.36 over every case here.
EL_FACTOR = 1.5


@pytest.fixture(scope="module")
def ec():
    from paper_2608_02474_gb300 import build
    build.build()
    from paper_2608_02474_gb300 import echocache
    echocache.lib()
    return echocache


def bf(a):
    return torch.from_numpy(np.ascontiguousarray(a, dtype=F32)).to(DEV, torch.bfloat16)


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


def check_active(g, o, emu, tag, mean_bar=5e-3):
    """Normwise and mean bars, and the element-wise figure against the model's."""
    mx, mean = normwise_rel(g, o)
    el = elementwise_rel(g, o)
    el_m = elementwise_rel(emu, o)
    print(f"[{tag}] rows {len(o)}: normwise {mx:.3e}  mean {mean:.3e}  elementwise {el:.3e}  "
          f"(ideal bf16 {el_m:.3e}, ratio {el / el_m:.2f})")
    assert mx <= 2e-2 and mean <= mean_bar, (tag, mx, mean, mean_bar)
    assert el <= EL_FACTOR * el_m, (tag, el, el_m)
    return mx, mean, el, el_m


def check_cache_and_inactive(ec, w, idx, q_in, s_in, g, y, gq, gs):
    """Inactive rows = the reconstructed cache, bit for bit; inactive cache rows
    untouched; the written cache rows = echo_cache_quant of the rows returned
    (echo_cache_quant is itself pinned bit-exact to the oracle)."""
    inactive = np.setdiff1d(np.arange(w.NT), idx)
    ref_inactive = oracle.cache.dequantize_rows(q_in[inactive], s_in[inactive])
    assert np.array_equal(g[inactive], ref_inactive)
    assert np.array_equal(gq[inactive], q_in[inactive]) and np.array_equal(gs[inactive], s_in[inactive])
    if len(idx):
        it = torch.from_numpy(idx.astype(np.int64)).to(DEV)
        q2 = torch.empty(len(idx), w.D, dtype=torch.int8, device=DEV)
        s2 = torch.empty(len(idx), dtype=torch.float32, device=DEV)
        ec.echo_cache_quant(y[it].contiguous(), None, q2, s2)
        assert np.array_equal(gq[idx], q2.cpu().numpy())
        assert np.array_equal(gs[idx], s2.cpu().numpy())


def check_layer(ec, w, res, q_in, s_in, g_idx, y, qd, sd, emu, tag, rows=None):
    assert np.array_equal(g_idx, res.idx)
    g = y.float().cpu().numpy()
    act = res.idx if rows is None else rows
    ya = res.y_act if rows is None else res.y_act_rows
    out = check_active(g[act], ya, emu, tag)
    check_cache_and_inactive(ec, w, res.idx, q_in, s_in, g, y, qd.cpu().numpy(), sd.cpu().numpy())
    return out


def _sample_rows(idx, scores, n=32, seed=0):
    """n rows of idx at random and the n of highest score (scores indexed by
    the values of idx), ascending and without repeats."""
    rng = np.random.default_rng(seed)
    top = idx[np.argsort(-scores[idx], kind="stable")[:n]]
    return np.unique(np.concatenate([rng.choice(idx, min(n, len(idx)), replace=False), top]))


def _trajectory(w, steps, layers, profile="speech"):
    audio = G.audio(w, profile)
    _, e = oracle.energy.audio_energy(audio, w.T)
    e32 = e.astype(F32)
    Ws = [G.block_weights(w, l) for l in range(layers)]
    cond = G.cond_tokens(w, audio)
    xs = list(G.step_inputs(w, G.latents(w), steps))
    rec = []
    oracle.step.generation(xs, Ws, [cond] * layers, e32, w.T, w.N, w.H, w.ratio_num, w.ratio_den,
                           record=lambda t, l, x, q, s, r: rec.append((t, l, x, q.copy(), s.copy(), r)))
    return Ws, cond, e32, rec


def _run_trajectory(ec, w, steps, layers, profile="speech", el_rows=256, mean_vs_model=False):
    """Every (step, layer) of the oracle's trajectory; all active rows at the
    normwise and mean bars, and up to `el_rows` of them (half at random, half
    of highest score) for the element-wise comparison with the model."""
    Ws, cond, e32, rec = _trajectory(w, steps, layers, profile)
    blks = [ec.DeviceBlock.from_host(W, cond) for W in Ws]
    for t, l, x, q, s, r in rec:
        g_idx, y, qd, sd = gpu_layer(ec, blks[l], w, x, q, s, e32, (w.ratio_num, w.ratio_den),
                                     full=t == 0)
        check_step(ec, w, Ws[l], cond, x, q, s, r, g_idx, y, qd, sd, f"{w.name} t={t} l={l}",
                   el_rows, mean_vs_model)


def check_step(ec, w, W, cond, x, q, s, r, g_idx, y, qd, sd, tag, el_rows=256,
               mean_vs_model=False):
    """One layer step against the oracle's result r on the same inputs: the
    indices, every active row at the normwise and mean bars, up to `el_rows`
    active rows (half at random, half of highest score) against the ideal bf16
    model element-wise, the inactive rows and the cache write.  mean_vs_model
    (rows wider than any of the paper's workloads, where the ideal bf16 block
    itself is above 5e-3): the mean bar is 1.25 times the model's mean on the
    same rows, every active row being compared with the model."""
    assert np.array_equal(g_idx, r.idx)
    g = y.float().cpu().numpy()
    mx, mean = normwise_rel(g[r.idx], r.y_act)
    j = np.arange(len(r.idx))
    if len(j) > el_rows:
        assert not mean_vs_model, "the model's mean needs every active row"
        j = _sample_rows(j, r.scores[r.idx], n=el_rows // 2)
    emu = M.block_active(x, r.idx[j], W, cond, w.H) if len(j) else None
    mean_bar = 5e-3
    if mean_vs_model and len(j):
        mean_bar = max(mean_bar, 1.25 * normwise_rel(emu, r.y_act[j])[1])
    assert mx <= 2e-2 and mean <= mean_bar, (tag, mx, mean, mean_bar)
    if len(j):
        check_active(g[r.idx[j]], r.y_act[j], emu, tag, mean_bar)
    check_cache_and_inactive(ec, w, r.idx, q, s, g, y, qd.cpu().numpy(), sd.cpu().numpy())


def test_tiny_every_step(ec):
    """The 256-token block over all 8 steps (step 0 full)."""
    _run_trajectory(ec, TINY_256, TINY_256.steps, TINY_256.layers)


def test_stack4_every_step(ec):
    """The 7800-token, 4-block stack over all 10 steps: from step 2 on the
    caches hold rows of different ages, and the selection decides which of them
    are refreshed."""
    _run_trajectory(ec, STACK4_7800, STACK4_7800.steps, STACK4_7800.layers)


@pytest.mark.parametrize("profile", ["silence", "tone", "beats"])
def test_tiny_profiles(ec, profile):
    _run_trajectory(ec, TINY_256, 3, 1, profile)


@pytest.mark.parametrize("H,d", [(64, 128), (128, 64)])
def test_widest_block_ragged_shapes(ec, H, d):
    """The widest rows the ABI takes (D 8192), every other size ragged: 70
    spatial latents per frame (210 tokens, divided by neither the 128-row
    attention tile nor the 256-row GEMM tile), an FFN of 1088 (4.25 GEMM
    N-tiles), 37 audio tokens (one masked key block), r = 1/3 (70 active
    rows); the full step and one cached step."""
    from dataclasses import replace
    w = replace(TINY_256, name=f"widest_{H}x{d}", T=3, Hp=7, Wp=10, D=8192, H=H, d=d, F=1088,
                Lc=37, n_samples=4800, ratio_num=1, ratio_den=3, steps=2, layers=1)
    # at this width the ideal bf16 block's own mean relative error is about
    # 8e-3 on these inputs (normwise max 1.1e-2): the mean is held against it
    _run_trajectory(ec, w, 2, 1, mean_vs_model=True)


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
    xd = bf(x)
    qd, sd = torch.from_numpy(q.copy()).to(DEV), torch.from_numpy(s.copy()).to(DEV)
    idx = torch.arange(w.NT, dtype=torch.int32, device=DEV)
    ec.echo_block_step(blk, dims, xd, idx, w.NT, qd, sd, y=xd)
    check_active(xd.float().cpu().numpy(), oracle.block.uncached_block(x, W, cond, w.H),
                 M.block_active(x, np.arange(w.NT), W, cond, w.H), "tiny K=NT aliased")
    assert ec.echo_get_device_error() == 0


@pytest.mark.parametrize("which", ["first", "last", "middle", "all_but_one"])
def test_one_active_row_and_all_but_one(ec, which):
    """K = 1 (one query row through every GEMM and both attentions) and
    K = NT - 1: an active row's output is the uncached block's at that row
    (K and V always cover every token), every other row is the reconstructed
    cache, and the cache holds the quantised rows returned."""
    w = TINY_256
    W = G.block_weights(w, 0)
    cond = G.cond_tokens(w, G.audio(w))
    x = G.latents(w)
    q, s = oracle.cache.quantize_rows(G.step_input(w, x, 2))[:2]
    blk = ec.DeviceBlock.from_host(W, cond)
    dims = ec.BlockDims(w.T, w.N, w.D, w.H, w.d, w.F, w.Lc)
    rows = {"first": [0], "last": [w.NT - 1], "middle": [w.NT // 2 + 3],
            "all_but_one": [i for i in range(w.NT) if i != 77]}[which]
    idx = np.asarray(rows, dtype=np.int32)
    qd, sd = torch.from_numpy(q.copy()).to(DEV), torch.from_numpy(s.copy()).to(DEV)
    y = ec.echo_block_step(blk, dims, bf(x), torch.from_numpy(idx).to(DEV), len(idx), qd, sd)
    torch.cuda.synchronize()
    assert ec.echo_get_device_error() == 0
    g = y.float().cpu().numpy()
    check_active(g[idx], oracle.block.uncached_block(x, W, cond, w.H)[idx],
                 M.block_active(x, idx, W, cond, w.H), f"tiny K={len(idx)} {which}")
    check_cache_and_inactive(ec, w, idx, q, s, g, y, qd.cpu().numpy(), sd.cpu().numpy())


# ---------------------------------------------------------------------------
# Full-size Wan2.2-S2V-shaped blocks (D 5120, 40 heads x 128, FFN 13824, 672
# audio tokens).  The oracle recomputes K/V over every token and the block for
# 64 sampled active rows: 32 at random and the 32 of highest score.



class _Sampled:
    """The oracle's sampled rows of one cached layer step."""

    def __init__(self, x, q, s, e32, w, W, cond, ratio, kv=None):
        self.idx, sc = oracle.select.select(x, q, s, e32, w.T, w.N, *ratio)
        self.rows = _sample_rows(self.idx, sc)
        Kv, Vv, Km, Vm = kv if kv is not None else (*oracle.block.self_kv(x, W),
                                                    *M.self_kv(x, W, fp32=True))
        Kc, Vc = oracle.block.cross_kv(cond, W)
        self.y_act_rows = oracle.block.active_rows(x, self.rows, W, w.H, Kv, Vv, Kc, Vc)
        self.emu = M.active_rows(x, self.rows, W, w.H, Km, Vm, *M.cross_kv(cond, W))


@pytest.mark.slow
def test_wan_block_sampled_rows(ec):
    """The 32760-token block at r = 1/5: step-1 input against the quantised
    step-0 latents, as after the full warm-up step."""
    w = WAN_BLOCK_32760
    audio = G.audio(w)
    e32 = oracle.energy.audio_energy(audio, w.T)[1].astype(F32)
    W = G.block_weights(w, 0)
    cond = G.cond_tokens(w, audio)
    x0 = G.latents(w)
    x1 = G.step_input(w, x0, 1)
    q, s, _ = oracle.cache.quantize_rows(x0)
    g_idx, y, qd, sd = gpu_layer(ec, ec.DeviceBlock.from_host(W, cond), w, x1, q, s, e32,
                                 (w.ratio_num, w.ratio_den))
    o = _Sampled(x1, q, s, e32, w, W, cond, (w.ratio_num, w.ratio_den))
    check_layer(ec, w, o, q, s, g_idx, y, qd, sd, o.emu, "wan_block_32760", rows=o.rows)


@pytest.fixture(scope="module")
def sweep_state():
    """63960-token block: the step-1 input, the cache of the quantised step-0
    latents, and the oracle's and the model's K/V over every token (these
    depend on neither the ratio nor the audio, so every case shares them)."""
    w = WAN_SWEEP_63960
    W = G.block_weights(w, 0)
    x0 = G.latents(w)
    x1 = G.step_input(w, x0, 1)
    q, s, _ = oracle.cache.quantize_rows(x0)
    del x0
    kv = (*oracle.block.self_kv(x1, W), *M.self_kv(x1, W, fp32=True))
    return w, W, x1, q, s, kv


@pytest.mark.slow
@pytest.mark.parametrize("profile,ratio", [("speech", (1, 20)), ("speech", (1, 10)),
                                           ("speech", (1, 5)), ("speech", (1, 2)),
                                           ("speech", (1, 1)), ("silence", (1, 5)),
                                           ("tone", (1, 5)), ("beats", (1, 5))],
                         ids=lambda v: v if isinstance(v, str) else f"r{v[0]}_{v[1]}")
def test_sweep_63960_sampled_rows(ec, sweep_state, profile, ratio):
    """The 161-frame sweep block (41 x 30 x 52 = 63960 tokens) at every ratio of
    the sweep with speech audio, and at r = 1/5 with the silence, tone and
    beats profiles (which change the segment weights and so the selection).
    r = 1/20 gives the thinnest attention grid (3198 queries), r = 1 refreshes
    every token."""
    w, W, x1, q, s, kv = sweep_state
    audio = G.audio(w, profile)
    e32 = oracle.energy.audio_energy(audio, w.T)[1].astype(F32)
    cond = G.cond_tokens(w, audio)
    g_idx, y, qd, sd = gpu_layer(ec, ec.DeviceBlock.from_host(W, cond), w, x1, q, s, e32, ratio)
    o = _Sampled(x1, q, s, e32, w, W, cond, ratio, kv=kv)
    assert len(o.idx) == oracle.select.refresh_budget(w.NT, *ratio)
    check_layer(ec, w, o, q, s, g_idx, y, qd, sd, o.emu,
                f"sweep_63960 {profile} r={ratio[0]}/{ratio[1]}", rows=o.rows)


@pytest.mark.slow
def test_stack40_gpu_trajectory(ec):
    """The 40-layer stack over 20 steps on the GPU's own trajectory
    (CachedStack: step 0 full, then r = 1/5 per step and per layer).  At steps
    {1, 10, 19} x layers {0, 19, 39} the GPU's layer input, its cache before the
    step and its segment energy are copied to the host and fed to the oracle:
    indices and inactive rows bit-exact, 64 sampled active rows at the bars.  By
    step 19 the cache holds rows written at many different steps, each with the
    scale the FFN-down epilogue's row maximum gave it."""
    from paper_2608_02474_gb300.pipeline import CachedStack
    w = WAN_STACK40_32760
    steps, check_steps, check_layers = w.steps, (1, 10, 19), (0, 19, 39)
    audio = G.audio(w)
    cond = G.cond_tokens(w, audio)
    blocks, Wk = [], {}
    for l in range(w.layers):
        W = G.block_weights(w, l)
        if l in check_layers:
            Wk[l] = W
        blocks.append(ec.DeviceBlock.from_host(W, cond))
        del W
    st = CachedStack(w.T, w.N, w.D, w.H, w.d, w.F, w.Lc, blocks, device=DEV)
    st.set_audio(torch.from_numpy(audio).to(DEV))
    st.wait_audio()
    e_gpu = st.seg.cpu().numpy().copy()
    e_ref = oracle.energy.audio_energy(audio, w.T)[1]
    assert np.all(np.abs(e_gpu - e_ref) <= 1e-5 * np.abs(e_ref))
    cur = {"t": 0}
    snap = {}
    done = []

    def hook(phase, l, x, idx, K, y):
        if cur["t"] not in check_steps or l not in check_layers:
            return
        if phase == "pre":
            torch.cuda.synchronize()
            snap["x"] = x.float().cpu().numpy()
            snap["q"] = st.cache_q[l].cpu().numpy()
            snap["s"] = st.cache_s[l].cpu().numpy()
            return
        torch.cuda.synchronize()
        assert ec.echo_get_device_error() == 0
        g_idx = idx[:K].cpu().numpy()
        o = _Sampled(snap["x"], snap["q"], snap["s"], e_gpu, w, Wk[l], cond,
                     (w.ratio_num, w.ratio_den))
        check_layer(ec, w, o, snap["q"], snap["s"], g_idx, y, st.cache_q[l], st.cache_s[l],
                    o.emu, f"stack40 t={cur['t']} l={l}", rows=o.rows)
        done.append((cur["t"], l))

    st.layer_hook = hook
    for t, x in enumerate(G.step_inputs(w, G.latents(w), steps)):
        cur["t"] = t
        st.step(bf(x), w.ratio_num, w.ratio_den, full=t == 0)
    torch.cuda.synchronize()
    assert ec.echo_get_device_error() == 0
    assert done == [(t, l) for t in check_steps for l in check_layers]


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
