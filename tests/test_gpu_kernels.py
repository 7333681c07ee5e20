"""GPU parity of each kernel entry point against the CPU oracle (same seeded inputs).

Bars: bit-exact for the int8 cache, scales, dequantised rows, drift scores and
selected indices; rel <= 1e-5 for fp32 energies; bf16 outputs within the
block tolerance (per-row normwise max rel <= 2e-2, mean rel <= 5e-3).
"""
import os

import numpy as np
import pytest
import torch

import oracle
from synth import ALL, generate as G

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ec():
    from paper_2608_02474_gb300 import build
    build.build()
    from paper_2608_02474_gb300 import echocache
    echocache.lib()
    return echocache


DEV = "cuda"
F32 = np.float32


def bf(a):
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(DEV, torch.bfloat16)


def f32(a):
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(DEV)


def close_bf16(g, o, max_rel=2e-2, mean_rel=5e-3):
    """Per-row normwise max relative error max_j|g-o| / max_j|o| and the mean
    relative error sum|g-o| / sum|o| (the reading justified in
    test_tolerance_reading.py)."""
    g = np.asarray(g, dtype=np.float64)
    o = np.asarray(o, dtype=np.float64)
    rel = np.abs(g - o).max(axis=-1) / np.maximum(np.abs(o).max(axis=-1), 1e-30)
    mr = np.abs(g - o).sum() / max(np.abs(o).sum(), 1e-30)
    assert rel.max() <= max_rel and mr <= mean_rel, (float(rel.max()), float(mr))
    return float(rel.max()), float(mr)


def no_device_error(ec):
    assert ec.echo_get_device_error() == 0


# ---------------------------------------------------------------- energy
@pytest.mark.parametrize("name", ["tiny_256", "stack4_7800", "wan_block_32760", "wan_sweep_63960"])
@pytest.mark.parametrize("profile", ["speech", "silence", "tone", "beats"])
def test_audio_energy(ec, name, profile):
    w = ALL[name]
    a = G.audio(w, profile)
    band, seg = ec.echo_audio_energy(f32(a), w.T)
    ob, oe = oracle.energy.audio_energy(a, w.T)
    g_seg, g_band = seg.cpu().numpy().astype(np.float64), band.cpu().numpy().astype(np.float64)
    if profile == "silence":
        assert (g_seg == 0).all() and (g_band == 0).all()
    else:
        assert (np.abs(g_seg - oe) <= 1e-5 * oe).all()
        floor = 1e-6 * oe.sum()
        assert (np.abs(g_band - ob) <= 1e-5 * ob + floor).all()
    no_device_error(ec)


def test_audio_energy_short_segments_and_other_fft(ec):
    g = np.random.default_rng(0)
    a = g.standard_normal(3000).astype(F32)
    # 64 .. 512 take the warp kernel (two frames per complex FFT), 1024 the
    # shared-memory kernel; odd frame counts leave a lone last frame
    for T, n_fft, hop, nb in ((10, 512, 160, 8), (3, 256, 100, 5), (2, 1024, 333, 3),
                              (5, 64, 20, 4), (2, 128, 50, 3), (1, 512, 160, 64)):
        band, seg = ec.echo_audio_energy(f32(a), T, n_fft, hop, nb)
        ob, oe = oracle.energy.audio_energy(a, T, n_fft, hop, nb)
        assert np.allclose(seg.cpu().numpy(), oe, rtol=1e-5, atol=0)
        assert np.allclose(band.cpu().numpy(), ob, rtol=1e-5, atol=1e-6 * oe.sum())


# ---------------------------------------------------------------- cache
@pytest.mark.parametrize("D", [8, 128, 1024, 5120])
@pytest.mark.parametrize("src_t", ["bf16", "f32"])
def test_quant_bit_exact(ec, D, src_t):
    n = 333
    v = G.random_rows(n, D, seed=D, scale=3.0)
    if src_t == "f32":
        v = (v * F32(1.0009765625)).astype(F32)     # values off the bf16 grid
    v[5] = 0.0
    v[7] *= F32(1e-30)
    v[9] *= F32(1e30)
    if src_t == "bf16":
        v = G.to_bf16_values(v)
    rows = np.random.default_rng(1).permutation(2 * n)[:n].astype(np.int32)
    q = torch.zeros(2 * n, D, dtype=torch.int8, device=DEV)
    s = torch.full((2 * n,), -1.0, dtype=torch.float32, device=DEV)
    src = bf(v) if src_t == "bf16" else f32(v)
    ec.echo_cache_quant(src, torch.from_numpy(rows).to(DEV), q, s)
    oq = np.zeros((2 * n, D), np.int8)
    os_ = np.full(2 * n, -1.0, F32)
    oracle.cache.quant_scatter(v, rows, oq, os_)
    assert np.array_equal(q.cpu().numpy(), oq)
    assert np.array_equal(s.cpu().numpy().view(np.uint32), os_.view(np.uint32))
    no_device_error(ec)


def test_quant_identity_rows_and_nonfinite_flag(ec):
    v = G.random_rows(40, 64, seed=3)
    v[11, 3] = np.inf
    q = torch.zeros(40, 64, dtype=torch.int8, device=DEV)
    s = torch.zeros(40, dtype=torch.float32, device=DEV)
    ec.echo_cache_quant(bf(v), None, q, s)
    assert ec.echo_get_device_error() == 5          # NONFINITE, then cleared
    assert ec.echo_get_device_error() == 0
    oq, os_, bad = oracle.cache.quantize_rows(v)
    assert bad[11] and not q[11].any() and np.isinf(s[11].item())
    ok = np.arange(40) != 11
    assert np.array_equal(q.cpu().numpy()[ok], oq[ok])
    assert np.array_equal(s.cpu().numpy()[ok], os_[ok])


@pytest.mark.parametrize("D", [16, 128, 5120])
@pytest.mark.parametrize("out_t", [torch.bfloat16, torch.float32])
def test_dequant_bit_exact(ec, D, out_t):
    q, s = G.random_cache(257, D, seed=D, zero_rows=3)
    rows = np.random.default_rng(2).integers(0, 257, size=100).astype(np.int32)
    out = ec.echo_cache_dequant(torch.from_numpy(q).to(DEV), f32(s), torch.from_numpy(rows).to(DEV),
                                dtype=out_t)
    c = (q[rows].astype(F32) * s[rows][:, None]).astype(F32)
    ref = oracle.cache.dequant_gather(q, s, rows) if out_t == torch.bfloat16 else c
    assert np.array_equal(out.float().cpu().numpy().view(np.uint32), ref.view(np.uint32))
    full = ec.echo_cache_dequant(torch.from_numpy(q).to(DEV), f32(s))
    assert np.array_equal(full.float().cpu().numpy(), oracle.cache.dequant_gather(q, s))


# ---------------------------------------------------------------- selection
SELECT_CASES = [
    # T, N, D, ratio, mode, distinct energies
    (4, 64, 128, (1, 4), 0, True),
    (4, 64, 128, (1, 4), 1, True),
    (4, 64, 128, (1, 4), 2, True),
    (3, 7, 64, (7, 9), 0, False),
    (5, 1560, 1024, (1, 5), 0, True),
    (5, 1560, 1024, (0, 1), 0, True),
    (5, 1560, 1024, (1, 1), 0, True),
    (2, 1000, 264, (1, 3), 0, False),
    (21, 1560, 5120, (1, 5), 0, True),
    (41, 1560, 128, (1, 20), 0, True),
    (1, 300, 64, (1, 4), 0, True),      # one audio segment: its weight is 1
    (1, 300, 64, (1, 4), 1, True),
]


@pytest.mark.parametrize("T,N,D,ratio,mode,distinct", SELECT_CASES)
def test_select_bit_exact(ec, T, N, D, ratio, mode, distinct):
    NT = T * N
    seed = T * 1000 + D
    x = G.random_rows(NT, D, seed=seed)
    q, s = G.random_cache(NT, D, seed=seed + 1, zero_rows=2)
    e = G.random_energy(T, seed=seed + 2, distinct=distinct)
    if not distinct:
        e[1] = e[0]
    xd = bf(x)
    scores = torch.empty(NT, dtype=torch.float32, device=DEV)
    idx, K, _ = ec.echo_select(xd, torch.from_numpy(q).to(DEV), f32(s), f32(e), T, N, *ratio,
                               mode=mode, scores=scores)
    oidx, osc = oracle.select.select(x, q, s, e, T, N, *ratio, mode=mode)
    assert K == len(oidx)
    assert np.array_equal(scores.cpu().numpy().view(np.uint32), osc.view(np.uint32))
    assert np.array_equal(idx.cpu().numpy(), oidx)
    # f32 input takes the same path
    idx2, _, _ = ec.echo_select(f32(x), torch.from_numpy(q).to(DEV), f32(s), f32(e), T, N, *ratio,
                                mode=mode)
    assert np.array_equal(idx2.cpu().numpy(), oidx)
    no_device_error(ec)


def test_select_ties_take_lowest_index(ec):
    T, N, D = 4, 300, 64
    x = np.ones((T * N, D), F32)
    q = np.zeros((T * N, D), np.int8)
    s = np.zeros(T * N, F32)
    e = np.ones(T, F32)
    idx, K, _ = ec.echo_select(bf(x), torch.from_numpy(q).to(DEV), f32(s), f32(e), T, N, 1, 3)
    assert list(idx.cpu().numpy()) == list(range(K))


def test_select_with_and_without_workspace_agree(ec):
    """Scores kept by the caller, in the workspace, or both: the same selection,
    equal to the oracle's, on a case with many equal scores (quantised energy,
    repeated rows)."""
    T, N, D = 21, 520, 128
    NT = T * N
    x = G.random_rows(NT, D, seed=41)
    x[::3] = x[0]
    q, s = G.random_cache(NT, D, seed=42)
    q[::3], s[::3] = q[0], s[0]
    e = np.floor(G.random_energy(T, seed=43) * 4).astype(F32)
    qd = torch.from_numpy(q).to(DEV)
    ws = torch.empty(ec.echo_select_workspace_size(T, N), dtype=torch.uint8, device=DEV)
    sc = torch.empty(NT, dtype=torch.float32, device=DEV)
    a, K, _ = ec.echo_select(bf(x), qd, f32(s), f32(e), T, N, 1, 5, scores=sc)
    b, _, _ = ec.echo_select(bf(x), qd, f32(s), f32(e), T, N, 1, 5, scores=sc, workspace=ws)
    c, _, _ = ec.echo_select(bf(x), qd, f32(s), f32(e), T, N, 1, 5, workspace=ws)
    oidx, _ = oracle.select.select(x, q, s, e, T, N, 1, 5)
    for r in (a, b, c):
        assert np.array_equal(r.cpu().numpy(), oidx)
    no_device_error(ec)


# Top-K alone (echo_select_random ranks caller keys): sizes around the split of
# the keys over the CTAs of the cluster kernel (10240 keys and up, slices of at
# most 51200 keys), the one-CTA kernel on either side, budgets of one key, of
# all but one, and inside a run of equal keys that crosses slices.
TOPK_SIZES = [(1, 4097), (1, 10239), (1, 10240), (1, 10241), (7, 4681), (21, 1560), (41, 1560),
              (1, 65536), (3, 100001), (1, 409600), (1, 409601)]


@pytest.mark.parametrize("T,N", TOPK_SIZES)
@pytest.mark.parametrize("keys_kind", ["uniform", "three_levels", "one_level", "signed"])
def test_topk_over_slices(ec, T, N, keys_kind):
    NT = T * N
    r = G.rng(NT + len(keys_kind))
    if keys_kind == "uniform":
        keys = r.random(NT, dtype=np.float32)
    elif keys_kind == "three_levels":   # ties at every budget below, across slices
        keys = np.floor(r.random(NT, dtype=np.float32) * 3).astype(F32)
    elif keys_kind == "one_level":
        keys = np.full(NT, 0.25, F32)
    else:                               # negative and positive keys
        keys = (r.random(NT, dtype=np.float32) - F32(0.5)) * F32(8)
        keys[keys == 0] = F32(1)
    kd = torch.from_numpy(keys).to(DEV)
    for num, den in ((1, NT), (1, 20), (1, 2), (NT - 1, NT)):
        idx, K = ec.echo_select_random(kd, T, N, num, den)
        torch.cuda.synchronize()
        assert K == oracle.select.refresh_budget(NT, num, den)
        assert np.array_equal(idx.cpu().numpy(), oracle.select.random_subset(keys, K)), (num, den)
    no_device_error(ec)


@pytest.mark.parametrize("NT", [65536, 10920, 409600])
def test_topk_first_call_in_a_process(ec, NT):
    """The first top-K of a process, at a size whose keys need more dynamic
    shared memory than the default cap leaves beside the kernel's own buffers."""
    import subprocess
    import sys
    code = (
        "import numpy as np, torch\n"
        "from paper_2608_02474_gb300 import echocache as ec\n"
        "import oracle\n"
        f"NT = {NT}\n"
        "keys = np.random.default_rng(NT).random(NT, dtype=np.float32)\n"
        "idx, K = ec.echo_select_random(torch.from_numpy(keys).cuda(), 1, NT, 1, 5)\n"
        "torch.cuda.synchronize()\n"
        "assert ec.echo_get_device_error() == 0\n"
        "assert np.array_equal(idx.cpu().numpy(), oracle.select.random_subset(keys, K))\n"
        "print('ok')\n")
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    r = subprocess.run([sys.executable, "-c", code], cwd=root, capture_output=True, text=True,
                       timeout=300)
    assert r.returncode == 0 and r.stdout.strip().endswith("ok"), r.stdout + r.stderr


def test_select_with_silence_is_drift_only(ec):
    T, N, D = 4, 64, 128
    x = G.random_rows(T * N, D, seed=5)
    q, s = G.random_cache(T * N, D, seed=6)
    e = np.zeros(T, F32)
    i0, _, _ = ec.echo_select(bf(x), torch.from_numpy(q).to(DEV), f32(s), f32(e), T, N, 1, 4)
    i2, _, _ = ec.echo_select(bf(x), torch.from_numpy(q).to(DEV), f32(s), f32(e), T, N, 1, 4,
                              mode=2)
    assert np.array_equal(i0.cpu().numpy(), i2.cpu().numpy())


# ---------------------------------------------------------------- layer norm
@pytest.mark.parametrize("D", [64, 128, 1024, 5120])
@pytest.mark.parametrize("in_t", ["bf16", "f32"])
def test_layernorm(ec, D, in_t):
    n = 77
    x = G.random_rows(n, D, seed=D + 7, scale=2.0) + F32(0.5)
    if in_t == "bf16":
        x = G.to_bf16_values(x)
    rows = np.random.default_rng(D).permutation(n)[:50].astype(np.int32)
    src = bf(x) if in_t == "bf16" else f32(x)
    out = ec.echo_layernorm(src, torch.from_numpy(rows).to(DEV))
    ref = oracle.block.layer_norm(x[rows])
    g = out.float().cpu().numpy()
    assert np.all(np.abs(g - ref) <= 2 ** -8 * np.abs(ref) + 2e-3)


@pytest.mark.parametrize("in_t", ["bf16", "f32"])
@pytest.mark.parametrize("n,D", [(1000, 64), (333, 1024), (1217, 5120), (90, 8192)])
def test_layernorm_all_rows(ec, n, D, in_t):
    """Every row (no gather): the bf16 form streams rows through shared memory
    by bulk copies; its bits equal those of the gathered form on the same rows."""
    x = G.random_rows(n, D, seed=D + n, scale=2.0) + F32(0.5)
    if in_t == "bf16":
        x = G.to_bf16_values(x)
    src = bf(x) if in_t == "bf16" else f32(x)
    out = ec.echo_layernorm(src)
    ref = oracle.block.layer_norm(x)
    g = out.float().cpu().numpy()
    assert np.all(np.abs(g - ref) <= 2 ** -8 * np.abs(ref) + 2e-3)
    if in_t == "bf16":
        rows = torch.arange(n, dtype=torch.int32, device=DEV)
        assert torch.equal(out, ec.echo_layernorm(src, rows))
    no_device_error(ec)


# ---------------------------------------------------------------- GEMM
GEMM_CASES = [
    # M, Kd, N
    (300, 192, 320),
    (128, 640, 256),
    (1, 64, 64),
    (1000, 1024, 1024),
    (513, 512, 128),
    (200, 5120, 512),
    # more 256 x 256 tiles than CTA pairs on the GPU: pairs take several tiles,
    # alternating their two accumulators, and the 6-stage ring wraps across tiles
    (2000, 64, 2560),
    (4100, 320, 1536),
]


@pytest.mark.parametrize("M,Kd,N", GEMM_CASES)
def test_linear_bias(ec, M, Kd, N):
    A = G.random_rows(M, Kd, seed=M + Kd)
    W = G.random_rows(N, Kd, seed=N + 1, scale=0.05)
    b = G.random_rows(1, N, seed=N + 2, scale=0.5)[0]
    out = ec.echo_linear(bf(A), bf(W), bf(b))
    ref = oracle.block.linear(A, W, b)
    close_bf16(out.float().cpu().numpy(), ref)
    no_device_error(ec)


def test_linear_gelu_and_residuals(ec):
    M, Kd, N = 333, 256, 384
    A = G.random_rows(M, Kd, seed=1)
    W = G.random_rows(N, Kd, seed=2, scale=0.08)
    b = G.random_rows(1, N, seed=3, scale=0.3)[0]
    lin = oracle.block.linear(A, W, b)
    g = ec.echo_linear(bf(A), bf(W), bf(b), act=1)
    close_bf16(g.float().cpu().numpy(), oracle.block.gelu_tanh(lin))
    # bf16 residual gathered by row index, fp32 output
    R = G.random_rows(1000, N, seed=4)
    rows = np.random.default_rng(5).permutation(1000)[:M].astype(np.int32)
    g = ec.echo_linear(bf(A), bf(W), bf(b), resid=bf(R), resid_rows=torch.from_numpy(rows).to(DEV),
                       out_dtype=torch.float32)
    ref = lin + R[rows]
    assert np.allclose(g.cpu().numpy(), ref, rtol=1e-4, atol=1e-4)
    # fp32 residual, bf16 output
    R2 = np.random.default_rng(6).standard_normal((M, N)).astype(F32)
    g = ec.echo_linear(bf(A), bf(W), bf(b), resid=f32(R2))
    close_bf16(g.float().cpu().numpy(), lin + R2)
    # no bias, strided A (a column slice of a wider matrix)
    wide = G.random_rows(M, 2 * Kd, seed=9)
    Ad = bf(wide)[:, Kd:]
    g = ec.echo_linear(Ad, bf(W))
    close_bf16(g.float().cpu().numpy(), wide[:, Kd:].astype(np.float64) @ W.T.astype(np.float64))
    no_device_error(ec)


# ---------------------------------------------------------------- attention
ATTN_CASES = [
    # M, L, H, d
    (200, 333, 2, 64),
    (200, 333, 2, 128),
    (1, 1, 1, 64),
    (128, 64, 4, 128),
    (130, 672, 3, 128),
    (64, 7800, 2, 64),
    # key sets up to 2048 take the persistent kernel (items chained per SM)
    (6552, 672, 40, 128),    # cross-attention of the 32760-token block: 1040 items, 96-key blocks
    (3000, 160, 16, 64),     # 192 items (some CTAs take two), 96-key blocks with a masked tail
    (1000, 64, 4, 128),      # 64-key blocks
    (300, 32, 3, 64),        # 32-key blocks
    (300, 2048, 2, 128),     # the largest key set of the persistent kernel
    (300, 2049, 2, 128),     # one key more: the one-shot kernel
    (300, 4096, 2, 64),
    (300, 4097, 2, 64),
]


@pytest.mark.parametrize("M,L,H,d", ATTN_CASES)
def test_attention(ec, M, L, H, d):
    D = H * d
    Q = G.random_rows(M, D, seed=M + d, scale=1.5)
    KV = G.random_rows(L, 2 * D, seed=L + d, scale=1.5)
    kvd = bf(KV)
    out = ec.echo_attention(bf(Q), kvd[:, :D], kvd[:, D:], H, d)
    ref = oracle.block.mha(Q.astype(np.float64), KV[:, :D].astype(np.float64),
                           KV[:, D:].astype(np.float64), H)
    close_bf16(out.float().cpu().numpy(), ref)
    no_device_error(ec)


@pytest.mark.parametrize("d", [64, 128])
def test_attention_running_max_jumps(ec, d):
    """Later key blocks whose logits exceed the first block's by far more than
    2^64 force the kernel's rescale path (running max refreshed, O and the row
    sum rescaled in tensor memory); the result must still match the oracle."""
    H, M, L = 2, 150, 700
    D = H * d
    g = np.random.default_rng(d)
    Q = np.full((M, D), 2.0, dtype=F32) + g.standard_normal((M, D)).astype(F32) * F32(0.05)
    K = g.standard_normal((L, D)).astype(F32) * F32(0.1)
    K[400:] += F32(3.0)                          # logits jump by ~ 6 d / sqrt(d) nats
    V = g.standard_normal((L, D)).astype(F32)
    Q, K, V = (G.to_bf16_values(a) for a in (Q, K, V))
    KV = np.concatenate([K, V], axis=1)
    kvd = bf(KV)
    out = ec.echo_attention(bf(Q), kvd[:, :D], kvd[:, D:], H, d)
    ref = oracle.block.mha(Q.astype(np.float64), K.astype(np.float64), V.astype(np.float64), H)
    close_bf16(out.float().cpu().numpy(), ref)
    no_device_error(ec)
