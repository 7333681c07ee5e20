"""echo_select_static: token selection that allocates no device memory.

Some callers cannot allocate device memory: code inside a host application
that reserves all device memory at start-up and forbids cudaMalloc afterwards,
or code on a latency-critical thread where cudaMalloc/cudaFree would
synchronise the device.  echo_select_static keeps its drift scores in a
library-owned static device array instead of a caller workspace.

The test calls it through the C ABI twice in a row, on different inputs and
sizes (the second call reuses the array the first one filled), and checks
that each call selects exactly the indices echo_select selects with a
workspace (indices are compared bit-exact, as in every selection test).
A third case at 63960 tokens, near the static array's limit (its keys split
over the 8-CTA cluster form of the top-K), is also compared with the oracle's
selection directly.
This file is collected last so that a failure here never hides another test.
"""
import ctypes

import numpy as np
import pytest
import torch

from synth import generate as G

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.fixture(scope="module")
def ec():
    from paper_2608_02474_gb300 import build
    build.build()
    from paper_2608_02474_gb300 import echocache
    echocache.lib()
    return echocache


def _inputs(T, N, D, seed):
    NT = T * N
    x = torch.from_numpy(G.random_rows(NT, D, seed=seed)).to(DEV, torch.bfloat16)
    q, s = G.random_cache(NT, D, seed=seed + 1, zero_rows=1)
    e = G.random_energy(T, seed=seed + 2)
    return (x, torch.from_numpy(q).to(DEV), torch.from_numpy(s).to(DEV),
            torch.from_numpy(e).to(DEV))


def _select_static(ec, x, q, s, e, T, N, ratio):
    L = ec.lib()
    idx = torch.full((T * N,), -1, dtype=torch.int32, device=DEV)
    K = ctypes.c_int32(-1)
    prm = ec.SelectParams(0.1, 1e-6, ec.MODE_ENERGY_DRIFT)
    st = L.echo_select_static(
        ctypes.c_void_p(x.data_ptr()), ec.ECHO_BF16, ctypes.c_void_p(q.data_ptr()),
        ctypes.c_void_p(s.data_ptr()), ctypes.c_void_p(e.data_ptr()), T, N, x.shape[1],
        ratio[0], ratio[1], ctypes.byref(prm), ctypes.c_void_p(idx.data_ptr()), ctypes.byref(K),
        ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert st == ec.ECHO_OK, ec.status_str(st)
    return idx[:K.value], K.value


def test_static_select_matches_workspace_select_on_two_calls(ec):
    # 32760 tokens (the Wan2.2-S2V-shaped block), then a smaller 256-token case
    for T, N, D, ratio, seed in ((21, 1560, 5120, (1, 5), 11), (4, 64, 128, (1, 4), 12)):
        x, q, s, e = _inputs(T, N, D, seed)
        got, K = _select_static(ec, x, q, s, e, T, N, ratio)
        ref, K_ref, _ = ec.echo_select(x, q, s, e, T, N, *ratio)
        torch.cuda.synchronize()
        assert K == K_ref
        assert np.array_equal(got.cpu().numpy(), ref.cpu().numpy())
    assert ec.echo_get_device_error() == 0


def test_static_select_near_the_size_limit_matches_the_oracle(ec):
    """41 x 1560 = 63960 tokens (the 161-frame sweep shape, at a small width),
    near the static array's 65536: more keys than one CTA holds in shared
    memory, split over the CTAs of the cluster top-K.  Two calls in a row
    (r = 1/20, then r = 1/2), each compared bit for bit with echo_select and
    with the oracle's selection."""
    import oracle
    T, N, D = 41, 1560, 64
    x, q, s, e = _inputs(T, N, D, 21)
    xh, qh, sh, eh = (t.float().cpu().numpy() if t.dtype == torch.bfloat16 else t.cpu().numpy()
                      for t in (x, q, s, e))
    for ratio in ((1, 20), (1, 2)):
        got, K = _select_static(ec, x, q, s, e, T, N, ratio)
        ref, K_ref, _ = ec.echo_select(x, q, s, e, T, N, *ratio)
        torch.cuda.synchronize()
        o_idx, _ = oracle.select.select(xh, qh, sh, eh, T, N, *ratio)
        assert K == K_ref == len(o_idx)
        assert np.array_equal(got.cpu().numpy(), ref.cpu().numpy())
        assert np.array_equal(got.cpu().numpy(), o_idx)
    assert ec.echo_get_device_error() == 0


def test_static_select_rejects_more_tokens_than_its_array(ec):
    x, q, s, e = _inputs(2, 64, 64, 13)
    idx = torch.empty(128, dtype=torch.int32, device=DEV)
    K = ctypes.c_int32(-1)
    prm = ec.SelectParams(0.1, 1e-6, 0)
    # 2 x 32769 tokens > 65536: refused before anything is enqueued
    st = ec.lib().echo_select_static(
        ctypes.c_void_p(x.data_ptr()), ec.ECHO_BF16, ctypes.c_void_p(q.data_ptr()),
        ctypes.c_void_p(s.data_ptr()), ctypes.c_void_p(e.data_ptr()), 2, 32769, 64, 1, 5,
        ctypes.byref(prm), ctypes.c_void_p(idx.data_ptr()), ctypes.byref(K), None)
    assert st == 3 and K.value == -1        # ECHO_ERR_WORKSPACE
