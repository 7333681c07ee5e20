"""GPU parity of the step-level adaptive update rate (Sec. 3.3 with Eq. 1).

echo_step_delta against the oracle's fp64 sums on the same seeded inputs (the
relative bound 1e-6 covers fp32 element differences, fp32 pairwise chunk sums
and a compensated fp32 running sum: a few units of 2^-24); echo_update_rate
bit-exact against the oracle's rule; the adaptive step loop teacher-forced
against the oracle's adaptive generation (every GPU call gets the oracle's
state, including the step outputs whose change decides the budget)."""
import math

import numpy as np
import pytest
import torch

import oracle
from oracle import schedule as S
from synth import STACK4_7800, TINY_256, WAN_BLOCK_32760, generate as G

pytestmark = pytest.mark.gpu
DEV = "cuda"
REL = 1e-6


@pytest.fixture(scope="module")
def ec():
    from paper_2608_02474_gb300 import build
    build.build()
    from paper_2608_02474_gb300 import echocache
    echocache.lib()
    return echocache


def _dev(a, bf16):
    return torch.from_numpy(np.ascontiguousarray(a)).to(DEV, torch.bfloat16 if bf16 else
                                                        torch.float32)


def _gpu_delta(ec, a, b, bf16=True, xi=1e-6):
    out = ec.echo_step_delta(_dev(a, bf16), _dev(b, bf16), xi)
    torch.cuda.synchronize()
    assert ec.echo_get_device_error() == 0
    return out.cpu().numpy()


def _close(g, o, rel=REL):
    return abs(g - o) <= rel * abs(o)


@pytest.mark.parametrize("bf16", [True, False])
@pytest.mark.parametrize("n", [1, 7, 8, 9, 4099, 256 * 128, 608 * 512 * 8 * 2 + 13, 7800 * 1024])
def test_step_delta_matches_oracle(ec, n, bf16):
    a, b = G.step_output_pair(n, seed=n % 1000, bf16=bf16)
    g = _gpu_delta(ec, a, b, bf16)
    num, den = S.step_sums(a, b)
    assert _close(g[1], num) and _close(g[2], den), (g, num, den)
    assert _close(g[0], S.step_delta(a, b), 2 * REL)


def test_step_delta_edge_cases(ec):
    # empty: all zero
    e = torch.empty(0, dtype=torch.bfloat16, device=DEV)
    out = ec.echo_step_delta(e, e)
    torch.cuda.synchronize()
    assert out.cpu().tolist() == [0.0, 0.0, 0.0]
    # identical outputs: no change at all, exactly
    a, _ = G.step_output_pair(100003, seed=5)
    g = _gpu_delta(ec, a, a)
    assert g[0] == 0.0 and g[1] == 0.0 and _close(g[2], S.step_sums(a, a)[1])
    # h_cur = 2 h_prev: every term of the second sum is exactly twice the
    # first one's, so the GPU's sums are in the ratio 2 bit for bit
    g = _gpu_delta(ec, a, 2 * a)
    assert g[2] == 2 * g[1] and _close(g[0], S.step_delta(a, 2 * a), 2 * REL)
    # all zero outputs: Delta = 0 / xi = 0
    z = np.zeros(4096, dtype=np.float32)
    assert _gpu_delta(ec, z, z).tolist() == [0.0, 0.0, 0.0]


def test_step_delta_is_deterministic(ec):
    a, b = G.step_output_pair(3_000_001, seed=9)
    da, db = _dev(a, True), _dev(b, True)
    outs = [ec.echo_step_delta(da, db).cpu().numpy().tobytes() for _ in range(3)]
    assert outs[0] == outs[1] == outs[2]


def test_step_delta_full_size(ec):
    """One output of the 32760-token, D = 5120 block (167.7M bf16 values)."""
    w = WAN_BLOCK_32760
    a, b = G.step_output_pair(w.NT * w.D, seed=31)
    g = _gpu_delta(ec, a, b)
    num, den = S.step_sums(a, b)
    assert _close(g[1], num) and _close(g[2], den), (g, num, den)
    assert _close(g[0], num / (den + 1e-6), 2 * REL)
    g2 = _gpu_delta(ec, a, 2 * a)
    assert g2[2] == 2 * g2[1]


def test_update_rate_matches_oracle_rule(ec):
    rs = np.random.default_rng(4)
    for _ in range(20000):
        d, ref = float(rs.uniform(0, 3)), float(rs.choice([0.0, rs.uniform(1e-3, 2)]))
        NT = int(rs.choice([1, 256, 7800, 32760, 63960]))
        r_min, r_max, alpha = 0.1, float(rs.choice([0.5, 1.0])), float(rs.choice([0.2, 0.35]))
        rate, K = ec.echo_update_rate(d, ref, NT, r_min, r_max, alpha)
        assert rate == S.update_rate(S.normalised(d, ref), r_min, r_max, alpha)
        assert K == S.adaptive_budget(d, ref, NT, r_min, r_max, alpha)


def _adaptive_trajectory(w, steps, layers, sch):
    audio = G.audio(w)
    _, e = oracle.energy.audio_energy(audio, w.T)
    e32 = e.astype(np.float32)
    Ws = [G.block_weights(w, l) for l in range(layers)]
    cond = G.cond_tokens(w, audio)
    x0 = G.latents(w)
    xs = [x0] + [G.step_input(w, x0, t) for t in range(1, steps)]
    rec = []
    oracle.step.generation(xs, Ws, [cond] * layers, e32, w.T, w.N, w.H, w.ratio_num, w.ratio_den,
                           record=lambda t, l, x, q, s, r: rec.append((t, l, x, q.copy(), s.copy(), r)),
                           rate=sch)
    return Ws, cond, e32, rec


@pytest.mark.parametrize("w,steps", [(TINY_256, TINY_256.steps), (STACK4_7800, 4)],
                         ids=["tiny_256", "stack4_7800"])
def test_adaptive_loop_teacher_forced(ec, w, steps):
    from test_gpu_block import check_step, gpu_layer
    sch = S.Schedule(w.NT)
    Ws, cond, e32, rec = _adaptive_trajectory(w, steps, w.layers, sch)
    last = w.layers - 1
    outs = [r.y_bf16 for t, l, x, q, s, r in rec if l == last]
    # the change of every consecutive pair of oracle step outputs
    g_delta = [_gpu_delta(ec, outs[t - 1], outs[t])[0] for t in range(1, steps)]
    for gd, od in zip(g_delta, sch.deltas):
        assert _close(gd, od, 2 * REL), (gd, od)
    # the budget of every cached step from the GPU's changes
    g_budget = []
    for t in range(1, steps):
        d, ref = (g_delta[t - 2], g_delta[0]) if t >= 2 else (1.0, 1.0)
        g_budget.append(ec.echo_update_rate(d, ref, w.NT)[1])
    assert g_budget == sch.budgets
    assert len(set(g_budget)) > 1 or steps <= 3
    blks = [ec.DeviceBlock.from_host(W, cond) for W in Ws]
    for t, l, x, q, s, r in rec:
        ratio = (w.ratio_num, w.ratio_den) if t == 0 else (g_budget[t - 1], w.NT)
        g_idx, y, qd, sd = gpu_layer(ec, blks[l], w, x, q, s, e32, ratio, full=t == 0)
        check_step(ec, w, Ws[l], cond, x, q, s, r, g_idx, y, qd, sd, f"adaptive {w.name} t={t} l={l}")


def _stack(ec, w):
    from paper_2608_02474_gb300.pipeline import CachedStack
    audio = G.audio(w)
    cond = G.cond_tokens(w, audio)
    blks = [ec.DeviceBlock.from_host(G.block_weights(w, l), cond) for l in range(w.layers)]
    st = CachedStack(w.T, w.N, w.D, w.H, w.d, w.F, w.Lc, blks)
    st.set_audio(torch.from_numpy(audio).to(DEV))
    x0 = G.latents(w)
    xs = [torch.from_numpy(x0).to(DEV, torch.bfloat16)] + [
        torch.from_numpy(G.step_input(w, x0, t)).to(DEV, torch.bfloat16) for t in range(1, w.steps)]
    return st, xs


def test_adaptive_stack_runs_the_rule(ec):
    """Free-running CachedStack with AdaptiveRate: every cached step's K is the
    rule applied to the change the stack itself measured."""
    from paper_2608_02474_gb300.pipeline import AdaptiveRate
    w = TINY_256
    st, xs = _stack(ec, w)
    rate = AdaptiveRate(w.NT)
    for t, x in enumerate(xs):
        st.step_adaptive(x, rate, full=t == 0)
        if t > 0:
            assert st.last_K == [rate.budgets[-1]] * w.layers
    torch.cuda.synchronize()
    assert ec.echo_get_device_error() == 0
    k1 = math.ceil(S.update_rate(1.0) * w.NT)
    assert rate.budgets[:2] == [k1, k1]
    assert len(rate.deltas) == len(xs) - 2 and all(d > 0 and math.isfinite(d) for d in rate.deltas)
    for t in range(3, len(xs)):
        # step t follows the change between the outputs of steps t-2 and t-1
        assert rate.budgets[t - 1] == ec.echo_update_rate(rate.deltas[t - 2], rate.deltas[0], w.NT)[1]
    lo, hi = math.ceil(0.1 * w.NT), math.ceil(0.5 * w.NT)
    assert all(lo <= k <= hi for k in rate.budgets)


def test_pinned_adaptive_rate_equals_fixed_ratio_on_gpu(ec):
    """r_min = r_max = 1/4: the adaptive stack is the fixed-ratio stack at 1/4,
    bit for bit (the same kernels on the same inputs)."""
    from paper_2608_02474_gb300.pipeline import AdaptiveRate
    w = TINY_256
    a, xs = _stack(ec, w)
    b, _ = _stack(ec, w)
    rate = AdaptiveRate(w.NT, 0.25, 0.25, 0.5)
    for t, x in enumerate(xs):
        ya = a.step_adaptive(x, rate, full=t == 0).clone()
        yb = b.step(x, 1, 4, full=t == 0).clone()
        assert torch.equal(ya, yb)
    assert rate.budgets == [64] * (len(xs) - 1)


def test_adaptive_host_buffers_match_device_steps(ec):
    from paper_2608_02474_gb300.pipeline import AdaptiveRate
    w = TINY_256
    a, xs = _stack(ec, w)
    b, _ = _stack(ec, w)
    ra, rb = AdaptiveRate(w.NT), AdaptiveRate(w.NT)
    a.step_adaptive(xs[0], ra, full=True)
    b.step_adaptive(xs[0], rb, full=True)
    ref = [a.step_adaptive(x, ra).clone() for x in xs[1:]]
    hx = [x.cpu().pin_memory() for x in xs[1:]]
    hy = [torch.empty_like(h).pin_memory() for h in hx]
    b.run_host(hx, hy, 1, 1, rate=rb)
    torch.cuda.synchronize()
    assert rb.budgets == ra.budgets
    for r, h in zip(ref, hy):
        assert torch.equal(r.cpu(), h)
