"""Failure detection, checkpoint/resume and profiling of the runtime around
the kernels (none of them has a counterpart in the paper)."""
import json
import os

import numpy as np
import pytest
import torch

from synth import TINY_256, generate as G

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.fixture(scope="module")
def ec():
    from paper_2608_02474_gb300 import build
    build.build()
    from paper_2608_02474_gb300 import echocache
    echocache.lib()
    return echocache


def test_bounded_wait_reports_timeout_and_context_survives(ec):
    """A wait on a barrier nothing completes gives up after 1 ms with
    ECHO_ERR_TIMEOUT; the flag clears on read and the context keeps working."""
    assert ec.echo_get_device_error() == 0
    ec.echo_check_timeout_path(1_000_000)
    assert ec.echo_get_device_error() == 6          # ECHO_ERR_TIMEOUT
    assert ec.echo_get_device_error() == 0          # cleared by the read
    x = torch.randn(64, 128, device=DEV).to(torch.bfloat16)
    y = ec.echo_layernorm(x)
    torch.cuda.synchronize()
    assert torch.isfinite(y.float()).all() and ec.echo_get_device_error() == 0
    with pytest.raises(ec.EchoError):
        ec.echo_check_timeout_path(10)              # limit below 1 us is refused


def _stack(ec, w, kind):
    from paper_2608_02474_gb300.pipeline import CachedStack
    audio = G.audio(w)
    cond = G.cond_tokens(w, audio)
    blks = [ec.DeviceBlock.from_host(G.block_weights(w, l), cond) for l in range(w.layers)]
    st = CachedStack(w.T, w.N, w.D, w.H, w.d, w.F, w.Lc, blks, cache_kind=kind, seg_len=8,
                     tau=0.5)
    st.set_audio(torch.from_numpy(audio).to(DEV))
    return st


@pytest.mark.parametrize("kind", [0, 2])
def test_cache_checkpoint_resume(ec, kind, tmp_path):
    """Save the caches after three steps, restore them into a fresh stack: the
    next step is the same bit for bit."""
    w = TINY_256
    x0 = G.latents(w)
    xs = [torch.from_numpy(x0 if t == 0 else G.step_input(w, x0, t)).to(DEV, torch.bfloat16)
          for t in range(5)]
    a = _stack(ec, w, kind)
    for t in range(3):
        a.step(xs[t], 1, 4, full=t == 0)
    path = str(tmp_path / "caches.pt")
    a.save_caches(path)
    b = _stack(ec, w, kind)
    b.load_caches(path)
    ya = a.step(xs[3], 1, 4).clone()
    yb = b.step(xs[3], 1, 4).clone()
    assert torch.equal(ya, yb)
    c = _stack(ec, w, 1 - kind if kind == 0 else 0)
    with pytest.raises(ValueError):
        c.load_caches(path)


def test_profile_report_from_env(ec, tmp_path, monkeypatch):
    out = tmp_path / "prof.json"
    monkeypatch.setenv("ECHO_PROFILE", str(out))
    w = TINY_256
    st = _stack(ec, w, 0)
    x = torch.from_numpy(G.latents(w)).to(DEV, torch.bfloat16)
    st.step(x, 1, 1, full=True)
    st.step(x, 1, 4)
    rep = st.profile_report()
    ec.echo_profile_enable(False)
    names = {k.split("[")[0] for k in rep}
    assert {"gemm_tcgen05", "attention", "drift_score", "topk_select", "merge_quant"} <= names
    assert json.loads(out.read_text()) == json.loads(json.dumps(rep))
    assert all(v["launches"] > 0 and v["ms"] >= 0 for v in rep.values())


@pytest.mark.parametrize("kind,selection", [(0, "energy"), (2, "energy"), (0, "uniform")])
def test_graph_replay_matches_eager_steps(ec, kind, selection):
    """A cached step captured as a CUDA graph and replayed on new inputs gives
    the same outputs and caches, bit for bit, as the same steps run eagerly."""
    from paper_2608_02474_gb300.pipeline import CachedStack
    from synth import STACK4_7800 as w
    audio = torch.from_numpy(G.audio(w)).to(DEV)
    cond = G.cond_tokens(w, G.audio(w))
    blks = [ec.DeviceBlock.from_host(G.block_weights(w, l), cond) for l in range(w.layers)]
    x0 = G.latents(w)
    xs = [torch.from_numpy(G.step_input(w, x0, t)).to(DEV, torch.bfloat16) for t in range(1, 6)]
    x0d = torch.from_numpy(x0).to(DEV, torch.bfloat16)
    stacks = []
    for _ in range(2):
        st = CachedStack(w.T, w.N, w.D, w.H, w.d, w.F, w.Lc, blks, cache_kind=kind, seg_len=w.Wp,
                         tau=0.5, selection=selection)
        st.set_audio(audio)
        st.step(x0d, 1, 1, full=True)
        st.step(xs[0], 1, 5)
        stacks.append(st)
    a, b = stacks
    xbuf = torch.empty_like(xs[0])
    ybuf = torch.empty_like(xs[0])
    g, y = a.capture_step(xbuf, 1, 5, out=ybuf)
    assert y.data_ptr() == ybuf.data_ptr()
    for x in xs[1:]:
        xbuf.copy_(x)
        g.replay()
        yb = b.step(x, 1, 5)
        torch.cuda.synchronize()
        assert torch.equal(ybuf, yb)
    ca, cb = a.cache_state(), b.cache_state()
    for la, lb in zip(ca["layers"], cb["layers"]):
        for n in la:
            assert torch.equal(la[n], lb[n]), n
    assert ec.echo_get_device_error() == 0
