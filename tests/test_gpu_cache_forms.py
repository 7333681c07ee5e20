"""GPU parity of the cache forms: the reference-plus-int8-residual manager of
Sec. 3.4 (ECHO_CACHE_REF) and the full-precision ablation form (ECHO_CACHE_BF16)
of Table 2, against the oracle's RefCache / FullCache.

Cache writes and reads are compared bit for bit (slots, reference counts,
codes, scales, reconstructions: every decision is taken in the same fp32
order on both sides).  The layer step is teacher-forced: every GPU step gets
the oracle's layer input and cache state; its output rows are held to the
normwise bars of test_gpu_block.py, and its cache write is checked against
echo_cache_write of the rows it returned."""
import numpy as np
import pytest
import torch

import oracle
from oracle import refcache as R
from synth import TINY_256, generate as G

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


def _bf(a):
    return torch.from_numpy(np.ascontiguousarray(a, dtype=F32)).to(DEV, torch.bfloat16)


def _rows(idx):
    return torch.from_numpy(np.asarray(idx, dtype=np.int32)).to(DEV)


def _same_state(ec, g, o):
    torch.cuda.synchronize()
    assert ec.echo_get_device_error() == 0
    assert np.array_equal(g.t["ref"].cpu().numpy(), o.ref)
    assert np.array_equal(g.t["q"].cpu().numpy(), o.q)
    assert np.array_equal(g.t["scale"].cpu().numpy(), o.s)
    if o.R_cap:
        assert np.array_equal(g.t["refcount"].cpu().numpy()[:o.R_cap], o.refcount)
        live = o.refcount > 0
        assert np.array_equal(g.t["pool"].float().cpu().numpy()[:o.R_cap][live], o.pool[live])
    assert np.array_equal(g.read().float().cpu().numpy(), o.reconstruct_bf16())
    assert g.stats() == o.stats()


@pytest.mark.parametrize("NT,D,R_cap,seg_len,tau,rho", [
    (256, 128, 256, 8, 0.9, 0.95),      # mixed references and residuals
    (416, 256, 416, 52, 0.8, 0.9),      # 52-token spatial rows
    (256, 128, 256, 8, 2.0, 0.95),      # every row a reference
    (256, 128, 256, 8, -2.0, 0.95),     # one reference per segment
    (256, 128, 40, 16, 0.95, 0.9),      # pool runs out: late runs fall back to plain int8
    (256, 128, 0, 8, 0.9, 0.95),        # no pool: the plain int8 cache
    (256, 128, 256, 1, 0.5, 0.95),      # unit segments
    (300, 64, 300, 300, 0.7, 0.8),      # one segment over every token
    (2048, 5120, 2048, 52, 0.9, 0.95),  # D of the 32760-token block
])
def test_ref_cache_writes_match_oracle(ec, NT, D, R_cap, seg_len, tau, rho):
    g = ec.DeviceCache(ec.CACHE_REF, NT, D, R_cap=R_cap, seg_len=seg_len, tau=tau)
    o = R.RefCache(NT, D, R_cap, seg_len, tau)
    rs = np.random.default_rng(NT + D + R_cap)
    for it in range(4):
        n = NT if it == 0 else int(rs.integers(1, NT + 1))
        rows = np.sort(rs.choice(NT, n, replace=False)).astype(np.int32)
        v = G.correlated_rows(n, D, seed=1000 * it + NT, rho=rho)
        g.write(_bf(v), _rows(rows))
        o.write(rows, v)
        _same_state(ec, g, o)
    # reading a subset returns the same rows
    sub = np.sort(rs.choice(NT, NT // 3, replace=False)).astype(np.int32)
    assert np.array_equal(g.read(_rows(sub)).float().cpu().numpy(), o.reconstruct_bf16()[sub])


def test_ref_cache_uses_both_forms(ec):
    """On correlated rows at tau = 0.9 both stored forms occur, and the residual
    form reconstructs closer than the plain int8 cache on the same rows."""
    NT, D = 512, 256
    v = G.correlated_rows(NT, D, seed=3, rho=0.97)
    g = ec.DeviceCache(ec.CACHE_REF, NT, D, seg_len=64, tau=0.9)
    p = ec.DeviceCache(ec.CACHE_INT8, NT, D)
    g.write(_bf(v), _rows(np.arange(NT)))
    p.write(_bf(v), _rows(np.arange(NT)))
    live, hw = g.stats()
    assert 8 <= live < NT // 2 and hw == live
    e_ref = (g.read().float() - _bf(v).float()).abs().sum().item()
    e_int8 = (p.read().float() - _bf(v).float()).abs().sum().item()
    assert e_ref < e_int8


def test_full_cache_write_read(ec):
    NT, D = 300, 64
    g = ec.DeviceCache(ec.CACHE_BF16, NT, D)
    o = R.FullCache(NT, D)
    rs = np.random.default_rng(5)
    for it in range(3):
        rows = np.sort(rs.choice(NT, 100, replace=False)).astype(np.int32)
        v = G.random_rows(100, D, seed=it)
        g.write(_bf(v), _rows(rows))
        o.write(rows, v)
        torch.cuda.synchronize()
        assert np.array_equal(g.read().float().cpu().numpy(), o.reconstruct_bf16())


@pytest.mark.parametrize("kind", ["bf16", "ref"])
def test_select_against_cache_forms(ec, kind):
    w = TINY_256
    x = G.step_input(w, G.latents(w), 2)
    prev = G.correlated_rows(w.NT, w.D, seed=9, rho=0.9)
    e = G.random_energy(w.T, seed=1)
    if kind == "bf16":
        g, o = ec.DeviceCache(ec.CACHE_BF16, w.NT, w.D), R.FullCache(w.NT, w.D)
    else:
        g = ec.DeviceCache(ec.CACHE_REF, w.NT, w.D, seg_len=8, tau=0.85)
        o = R.RefCache(w.NT, w.D, w.NT, 8, 0.85)
    rows = np.arange(w.NT, dtype=np.int32)
    g.write(_bf(prev), _rows(rows))
    o.write(rows, prev)
    for mode in (0, 2):
        sc = torch.empty(w.NT, dtype=torch.float32, device=DEV)
        idx, K, _ = ec.echo_select_cache(_bf(x), g, torch.from_numpy(e).to(DEV), w.T, w.N, 1, 4,
                                         mode=mode, scores=sc)
        torch.cuda.synchronize()
        ref_sc = oracle.select.scores_from(x, o.reconstruct_f32(), e, w.T, w.N, mode=mode)
        assert np.array_equal(sc.cpu().numpy(), ref_sc)
        assert np.array_equal(idx.cpu().numpy(), oracle.select.top_k(ref_sc, K))


def _device_cache_from(ec, o, w):
    if o.kind == "bf16":
        g = ec.DeviceCache(ec.CACHE_BF16, w.NT, w.D)
        g.load(full=o.v)
    else:
        g = ec.DeviceCache(ec.CACHE_REF, w.NT, w.D, R_cap=o.R_cap, seg_len=o.seg_len,
                           tau=float(o.tau))
        g.load(q=o.q, scale=o.s, ref=o.ref)
        if o.R_cap:
            g.load(pool=o.pool, refcount=o.refcount)
    return g


@pytest.mark.parametrize("kind", ["bf16", "ref"])
def test_layer_step_with_cache_forms_teacher_forced(ec, kind):
    from bf16_model import normwise_rel as rel_err
    w = TINY_256
    audio = G.audio(w)
    _, e = oracle.energy.audio_energy(audio, w.T)
    e32 = e.astype(F32)
    W, cond = G.block_weights(w, 0), G.cond_tokens(w, audio)
    blk = ec.DeviceBlock.from_host(W, cond)
    dims = ec.BlockDims(w.T, w.N, w.D, w.H, w.d, w.F, w.Lc)
    x0 = G.latents(w)
    o = R.FullCache(w.NT, w.D) if kind == "bf16" else R.RefCache(w.NT, w.D, w.NT, 8, 0.0)
    for t in range(5):
        x = x0 if t == 0 else G.step_input(w, x0, t)
        res = oracle.step.cached_layer_step_cache(x, o, e32, W, cond, w.T, w.N, w.H, 1, 4,
                                                  full=t == 0)
        g = _device_cache_from(ec, o, w)
        before = g.clone()
        if t == 0:
            idx, K = torch.arange(w.NT, dtype=torch.int32, device=DEV), w.NT
        else:
            idx, K, _ = ec.echo_select_cache(_bf(x), g, torch.from_numpy(e32).to(DEV), w.T, w.N,
                                             1, 4)
        y = ec.echo_block_step_cache(blk, dims, _bf(x), idx, K, g)
        torch.cuda.synchronize()
        assert ec.echo_get_device_error() == 0
        gi = idx.cpu().numpy()
        assert np.array_equal(gi, res.idx)
        gy = y.float().cpu().numpy()
        mx, mean = rel_err(gy[gi], res.y_act)
        assert mx <= 2e-2 and mean <= 5e-3, (mx, mean)
        inactive = np.setdiff1d(np.arange(w.NT), gi)
        assert np.array_equal(gy[inactive], o.reconstruct_bf16()[inactive])
        # the step's cache write == echo_cache_write of the rows it returned
        before.write(y[idx.long()].contiguous(), idx)
        torch.cuda.synchronize()
        for n in g.t:
            assert torch.equal(g.t[n], before.t[n]), n
        o = res.cache


@pytest.mark.slow
def test_ref_cache_block_full_size_sampled(ec):
    """The 32760-token block (D 5120, 40 heads, r = 1/5) with the reference
    cache (tau 0.9, segments of 52 tokens) on spatially smooth latents: the
    oracle's cache state is loaded, indices and inactive rows are bit-exact,
    64 sampled active rows are held to the normwise bars, and the cache write
    equals echo_cache_write of the rows the step returned."""
    from synth import WAN_BLOCK_32760 as w
    from bf16_model import normwise_rel as rel_err
    audio = G.audio(w)
    _, e = oracle.energy.audio_energy(audio, w.T)
    e32 = e.astype(F32)
    W, cond = G.block_weights(w, 0), G.cond_tokens(w, audio)
    x0 = G.latents_smooth(w)
    x1 = G.step_input(w, x0, 1)
    o = R.RefCache(w.NT, w.D, w.NT, w.Wp, 0.9)
    o.write(np.arange(w.NT), x0)
    live, hw = o.stats()
    assert 0 < live < w.NT
    g = _device_cache_from(ec, o, w)
    before = g.clone()
    blk = ec.DeviceBlock.from_host(W, cond)
    dims = ec.BlockDims(w.T, w.N, w.D, w.H, w.d, w.F, w.Lc)
    xd = _bf(x1)
    idx, K, _ = ec.echo_select_cache(xd, g, torch.from_numpy(e32).to(DEV), w.T, w.N, 1, 5)
    y = ec.echo_block_step_cache(blk, dims, xd, idx, K, g)
    torch.cuda.synchronize()
    assert ec.echo_get_device_error() == 0
    sc = oracle.select.scores_from(x1, o.reconstruct_f32(), e32, w.T, w.N)
    oidx = oracle.select.top_k(sc, K)
    gi = idx.cpu().numpy()
    assert np.array_equal(gi, oidx)
    gy = y.float().cpu().numpy()
    inactive = np.setdiff1d(np.arange(w.NT), gi)
    assert np.array_equal(gy[inactive], o.reconstruct_bf16()[inactive])
    rng = np.random.default_rng(0)
    top = oidx[np.argsort(-sc[oidx], kind="stable")[:32]]
    rows = np.unique(np.concatenate([rng.choice(oidx, 32, replace=False), top]))
    Kv, Vv = oracle.block.self_kv(x1, W)
    Kc, Vc = oracle.block.cross_kv(cond, W)
    ya = oracle.block.active_rows(x1, rows, W, w.H, Kv, Vv, Kc, Vc)
    mx, mean = rel_err(gy[rows], ya)
    assert mx <= 2e-2 and mean <= 5e-3, (mx, mean)
    before.write(y[idx.long()].contiguous(), idx)
    torch.cuda.synchronize()
    for n in g.t:
        assert torch.equal(g.t[n], before.t[n]), n


@pytest.mark.parametrize("kind", ["bf16", "ref"])
def test_layer_step_with_no_active_rows(ec, kind):
    """K = 0: the step returns the cache's reconstruction and leaves the cache
    as it was."""
    w = TINY_256
    W, cond = G.block_weights(w, 0), G.cond_tokens(w, G.audio(w))
    blk = ec.DeviceBlock.from_host(W, cond)
    dims = ec.BlockDims(w.T, w.N, w.D, w.H, w.d, w.F, w.Lc)
    v = G.correlated_rows(w.NT, w.D, seed=12, rho=0.9)
    if kind == "bf16":
        g = ec.DeviceCache(ec.CACHE_BF16, w.NT, w.D)
    else:
        g = ec.DeviceCache(ec.CACHE_REF, w.NT, w.D, seg_len=8, tau=0.8)
    g.write(_bf(v), _rows(np.arange(w.NT)))
    before = g.clone()
    x = _bf(G.latents(w))
    y = ec.echo_block_step_cache(blk, dims, x, None, 0, g)
    torch.cuda.synchronize()
    assert ec.echo_get_device_error() == 0
    assert torch.equal(y, g.read())
    for n in g.t:
        assert torch.equal(g.t[n], before.t[n]), n
