"""GPU parity of the ablation modes of Sec. 4 (Table 2): Uniform and Random
selection in place of the energy-guided anchors, bit-exact against the oracle."""
import numpy as np
import pytest
import torch

from oracle import select as S
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


@pytest.mark.parametrize("T,N,num,den", [(4, 64, 1, 4), (21, 1560, 1, 5), (41, 1560, 1, 20),
                                         (5, 1560, 0, 1), (5, 1560, 1, 1), (3, 7, 2, 3)])
def test_uniform_selection(ec, T, N, num, den):
    idx, K = ec.echo_select_uniform(T, N, num, den)
    torch.cuda.synchronize()
    assert K == S.refresh_budget(T * N, num, den)
    assert np.array_equal(idx.cpu().numpy(), S.uniform(T * N, K))


@pytest.mark.parametrize("T,N,num,den,levels", [(4, 64, 1, 4, 0), (21, 1560, 1, 5, 0),
                                                (41, 1560, 1, 10, 0), (21, 1560, 1, 5, 7),
                                                (2, 5, 3, 5, 2)])
def test_random_selection(ec, T, N, num, den, levels):
    keys = G.rng(T * N + levels).random(T * N, dtype=np.float32)
    if levels:                     # many equal keys: ties go to the lower index
        keys = np.floor(keys * levels).astype(np.float32)
    idx, K = ec.echo_select_random(torch.from_numpy(keys).to(DEV), T, N, num, den)
    torch.cuda.synchronize()
    assert K == S.refresh_budget(T * N, num, den)
    assert np.array_equal(idx.cpu().numpy(), S.random_subset(keys, K))
