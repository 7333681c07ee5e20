"""The C-ABI library: it builds, loads, exports every declared symbol, and its
host-side argument checks reject bad calls before anything reaches a GPU."""
import ctypes
import glob
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def ec():
    import shutil
    if not shutil.which("nvcc") and not os.path.exists("/usr/local/cuda/bin/nvcc"):
        pytest.skip("nvcc not available")
    from paper_2608_02474_gb300 import build
    build.build()
    from paper_2608_02474_gb300 import echocache
    return echocache


def declared_functions():
    names = set()
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        src = open(h).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        for m in re.finditer(r"^[A-Za-z_][\w\s\*]*?\b(echo_\w+)\s*\(", src, flags=re.M):
            names.add(m.group(1))
    return sorted(names)


def test_header_declares_the_boundary():
    names = declared_functions()
    for n in ("echo_audio_energy", "echo_select", "echo_block_step", "echo_cache_quant",
              "echo_cache_dequant", "echo_precompute_cross_kv", "echo_workspace_size",
              "echo_get_device_error", "echo_status_str"):
        assert n in names


def test_every_declared_symbol_is_exported(ec):
    L = ctypes.CDLL(ec.LIB_PATH)
    missing = [n for n in declared_functions() if not hasattr(L, n)]
    assert not missing, missing


def test_binding_covers_every_symbol(ec):
    assert set(declared_functions()) <= set(ec._SIGS)


def test_status_strings(ec):
    assert ec.status_str(0) == "ECHO_OK"
    assert ec.status_str(3) == "ECHO_ERR_WORKSPACE"
    assert ec.status_str(99) == "ECHO_ERR_UNKNOWN"


FAKE = 0x10000  # a 16-byte aligned address that is never dereferenced by the checks


def _vp(v):
    return ctypes.c_void_p(v)


def test_select_argument_checks(ec):
    L = ec.lib()
    prm = ec.SelectParams(0.1, 1e-6, 0)
    K = ctypes.c_int32(-1)
    call = lambda x=FAKE, T=4, N=64, D=128, rn=1, rd=4, ws=FAKE, wsb=1 << 20, p=prm: L.echo_select(
        _vp(x), 0, _vp(FAKE), _vp(FAKE), _vp(FAKE), T, N, D, rn, rd, ctypes.byref(p), _vp(FAKE),
        ctypes.byref(K), None, _vp(ws), wsb, None)
    assert call(x=0) == 1                       # null
    assert call(x=FAKE + 2) == 1                # misaligned
    assert call(D=100) == 2                     # D % 8
    assert call(rn=5, rd=4) == 2                # ratio > 1
    assert call(rd=0) == 2
    assert call(wsb=16) == 3                    # workspace too small
    assert call(p=ec.SelectParams(0.1, 0.0, 0)) == 1   # xi must be > 0
    assert call(p=ec.SelectParams(0.1, 1e-6, 7)) == 1  # bad mode
    assert K.value == -1                        # nothing was written on failure


def test_block_step_argument_checks(ec):
    L = ec.lib()
    dims = ec.BlockDims(4, 64, 128, 2, 64, 512, 32)
    w = ec.BlockWeightsC(*([FAKE] * 15))
    ws = ec.echo_workspace_size(dims, 64)
    assert ws > 0
    call = lambda d=dims, K=64, wsb=ws, x=FAKE, w_=w: L.echo_block_step(
        ctypes.byref(w_), ctypes.byref(d), _vp(x), _vp(FAKE), K, _vp(FAKE), _vp(FAKE), _vp(FAKE),
        _vp(FAKE), wsb, None)
    assert call(d=ec.BlockDims(4, 64, 128, 2, 32, 512, 32)) == 2   # head size 32
    assert call(d=ec.BlockDims(4, 64, 128, 3, 64, 512, 32)) == 2   # H d != D
    assert call(K=257) == 2                                        # K > NT
    assert call(K=-1) == 2
    assert call(wsb=ws - 1) == 3
    assert call(x=FAKE + 8) == 1
    assert call(w_=ec.BlockWeightsC(*([FAKE] * 14 + [0]))) == 1     # null KVc


def test_block_step_kv_argument_checks(ec):
    """echo_block_step_kv: every check answers before anything is enqueued."""
    L = ec.lib()
    dims = ec.BlockDims(4, 64, 128, 2, 64, 512, 32)
    w = ec.BlockWeightsC(*([FAKE] * 15))
    ws = ec.echo_workspace_size_kv(dims, 64, 40)
    assert ws > 0
    call = lambda K=64, kv=FAKE, valid=1, ra=FAKE, na=20, rb=FAKE, nb=20, wsb=ws: L.echo_block_step_kv(
        ctypes.byref(w), ctypes.byref(dims), _vp(FAKE), _vp(FAKE), K, _vp(kv), valid, _vp(ra), na,
        _vp(rb), nb, _vp(FAKE), _vp(FAKE), _vp(FAKE), _vp(FAKE), wsb, None)
    assert call(kv=0) == 1                       # no K/V buffer
    assert call(kv=FAKE + 8) == 1                # misaligned K/V buffer
    assert call(na=-1) == 2
    assert call(ra=0) == 1                       # rows listed but no list
    assert call(ra=FAKE + 4) == 1
    assert call(K=257) == 2
    assert call(wsb=4096) == 3                   # far below 64 active, 40 recomputed rows
    # more rows need more workspace; kv_valid = 0 ignores the lists
    assert ec.echo_workspace_size_kv(dims, 64, 41) >= ws
    assert call(valid=0, ra=0, na=-5, wsb=ec.echo_workspace_size_kv(dims, 64, 0) - 1) == 3


def test_workspace_size_kv_leaves_kv_to_the_caller(ec):
    dims = ec.BlockDims(21, 1560, 5120, 40, 128, 13824, 672)
    NT, D = 32760, 5120
    plain = ec.echo_workspace_size(dims, 6552)
    kept = ec.echo_workspace_size_kv(dims, 6552, NT)
    # the all-token K/V (NT x 2D bf16) lives in the caller's buffer instead
    assert plain - kept >= 4 * NT * D - 4 * NT - 4096
    assert ec.echo_workspace_size_kv(dims, 6552, 13104) <= kept


def test_workspace_size_grows_with_K(ec):
    dims = ec.BlockDims(21, 1560, 5120, 40, 128, 13824, 672)
    a, b = ec.echo_workspace_size(dims, 0), ec.echo_workspace_size(dims, 6552)
    assert 0 < a < b
    NT, D, F, K = 32760, 5120, 13824, 6552
    # every buffer is at least its payload: n1, kv, rowmap plus the K-row buffers
    assert b >= 2 * NT * D + 4 * NT * D + 4 * NT + K * D * (2 * 4 + 4 * 2) + 2 * K * F
    assert ec.echo_select_workspace_size(21, 1560) >= 4 * 32760


def test_kernel_entry_points_check_shapes(ec):
    L = ec.lib()
    # echo_linear: Kd not a multiple of 64
    assert L.echo_linear(_vp(FAKE), 100, 8, 100, _vp(FAKE), None, 64, 0, None, 0, None, _vp(FAKE),
                         64, 0, None) == 2
    # echo_attention: head size 96
    assert L.echo_attention(_vp(FAKE), 192, _vp(FAKE), _vp(FAKE), 192, 4, 4, 2, 96, _vp(FAKE), 192,
                            None) == 2
    # echo_layernorm: D not a multiple of 8
    assert L.echo_layernorm(_vp(FAKE), 0, None, 4, 12, _vp(FAKE), None) == 2
    # echo_cache_dequant: D not a multiple of 16
    assert L.echo_cache_dequant(_vp(FAKE), _vp(FAKE), None, 4, 24, _vp(FAKE), 0, None) == 2
    # echo_audio_energy: n_fft not a power of two
    assert L.echo_audio_energy(_vp(FAKE), 16000, 4, 500, 160, 8, _vp(FAKE), _vp(FAKE), None) == 2
    # zero rows are a no-op
    assert L.echo_cache_quant(None, 0, None, 0, 64, None, None, None) == 0


def test_step_delta_argument_checks(ec):
    L = ec.lib()
    out = ctypes.c_void_p(FAKE)
    ws = ec.echo_step_delta_workspace_size(1 << 20)
    assert ws >= 16
    call = lambda a=FAKE, n=1024, xi=1e-6, wsb=ws, o=FAKE, dt=0: L.echo_step_delta(
        _vp(a), _vp(FAKE), dt, n, xi, _vp(o), _vp(FAKE), wsb, None)
    assert call(a=0) == 1                      # null input
    assert call(a=FAKE + 2) == 1               # misaligned
    assert call(o=FAKE + 4) == 1               # misaligned double output
    assert call(dt=5) == 1                     # unknown dtype
    assert call(xi=0.0) == 1                   # xi must be > 0
    assert call(n=-1) == 2
    assert call(wsb=ws - 1) == 3


def test_update_rate_rule_is_the_oracle_rule(ec):
    """echo_update_rate is host arithmetic: its rate and budget are those of the
    oracle's rule for the same change, bit for bit."""
    import numpy as np
    from oracle import schedule as S
    rs = np.random.default_rng(11)
    for _ in range(20000):
        d, ref = float(rs.uniform(0, 3)), float(rs.choice([0.0, rs.uniform(1e-3, 2)]))
        NT = int(rs.choice([0, 1, 256, 7800, 32760, 63960]))
        r_min = float(rs.choice([0.0, 0.05, 0.1]))
        r_max, alpha = float(rs.choice([0.3, 0.5, 1.0])), float(rs.choice([0.0, 0.2, 0.35, 1e6]))
        rate, K = ec.echo_update_rate(d, ref, NT, r_min, r_max, alpha)
        assert rate == S.update_rate(S.normalised(d, ref), r_min, r_max, alpha)
        assert K == S.adaptive_budget(d, ref, NT, r_min, r_max, alpha)
    # the clip and the first cached step (Delta-hat = 1)
    assert ec.echo_update_rate(0.0, 1.0, 100) == (0.1, 10)
    assert ec.echo_update_rate(9.0, 1.0, 100) == (0.5, 50)
    with pytest.raises(ec.EchoError):
        ec.echo_update_rate(float("nan"), 1.0, 100)
    with pytest.raises(ec.EchoError):
        ec.echo_update_rate(0.1, 1.0, 100, r_min=0.6, r_max=0.5)


def test_ablation_selection_argument_checks(ec):
    L = ec.lib()
    K = ctypes.c_int32(-1)
    assert L.echo_select_uniform(4, 64, 1, 4, None, ctypes.byref(K), None) == 1
    assert L.echo_select_uniform(4, 64, 5, 4, _vp(FAKE), ctypes.byref(K), None) == 2
    assert L.echo_select_uniform(0, 64, 1, 4, _vp(FAKE), ctypes.byref(K), None) == 2
    assert L.echo_select_random(_vp(FAKE + 4), 4, 64, 1, 4, _vp(FAKE), ctypes.byref(K), None) == 1
    assert L.echo_select_random(_vp(FAKE), 4, 64, 1, 0, _vp(FAKE), ctypes.byref(K), None) == 2
    assert K.value == -1


def test_cache_form_argument_checks(ec):
    L = ec.lib()
    mk = lambda kind=2, NT=64, D=64, ref=FAKE, R_cap=64, seg=8: ec.CacheC(
        kind, NT, D, FAKE, FAKE, FAKE, ref, FAKE, FAKE, R_cap, seg, 0.9)
    c = mk()
    assert ec.lib().echo_cache_write_workspace_size(ctypes.byref(c), 64) > 0
    assert L.echo_cache_write(ctypes.byref(mk(kind=7)), _vp(FAKE), _vp(FAKE), 4, _vp(FAKE),
                              1 << 20, None) == 1
    assert L.echo_cache_write(ctypes.byref(mk(D=24)), _vp(FAKE), _vp(FAKE), 4, _vp(FAKE),
                              1 << 20, None) == 2
    assert L.echo_cache_write(ctypes.byref(mk(ref=0)), _vp(FAKE), _vp(FAKE), 4, _vp(FAKE),
                              1 << 20, None) == 1
    assert L.echo_cache_write(ctypes.byref(mk(seg=0)), _vp(FAKE), _vp(FAKE), 4, _vp(FAKE),
                              1 << 20, None) == 1
    assert L.echo_cache_write(ctypes.byref(c), _vp(FAKE), _vp(FAKE), 65, _vp(FAKE),
                              1 << 20, None) == 2
    assert L.echo_cache_write(ctypes.byref(c), _vp(FAKE), _vp(FAKE), 4, _vp(FAKE), 16, None) == 3
    assert L.echo_cache_write(ctypes.byref(c), _vp(FAKE), _vp(FAKE), 0, None, 0, None) == 0
    assert L.echo_cache_stats(ctypes.byref(mk(kind=1)), _vp(FAKE), None) == 1
    dims = ec.BlockDims(4, 16, 64, 1, 64, 128, 8)
    w = ec.BlockWeightsC(*([FAKE] * 15))
    # the cache must match the block's NT and D
    assert L.echo_block_step_cache(ctypes.byref(w), ctypes.byref(dims), _vp(FAKE), _vp(FAKE), 4,
                                   ctypes.byref(mk(NT=65)), _vp(FAKE), _vp(FAKE), 1 << 30,
                                   None) == 2


def test_timeout_probe_argument_checks(ec):
    L = ec.lib()
    assert L.echo_check_timeout_path(999, None) == 1
    assert L.echo_check_timeout_path(3_000_000_000, None) == 1
