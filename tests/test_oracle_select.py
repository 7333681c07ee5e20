"""Pins for the oracle's per-token drift (Eq. 1) and the energy-weighted selection (Sec. 3.3)."""
import itertools
import math

import numpy as np
import pytest

from oracle import select as S
from synth import generate as G

F32 = np.float32


def test_canonical_order_within_a_chunk_is_left_to_right():
    # 2^24 + 1 + 1 summed left to right loses both ones (ties to even); a pairwise
    # or reversed order would keep them.
    v = np.zeros((1, 8), dtype=F32)
    v[0, :3] = [2.0 ** 24, 1.0, 1.0]
    assert S.canonical_sum(v)[0] == F32(2.0 ** 24)
    v[0, :3] = [1.0, 1.0, 2.0 ** 24]
    assert S.canonical_sum(v)[0] == F32(2.0 ** 24 + 2)


def test_canonical_order_lanes_then_butterfly():
    # D = 512: 64 chunks; lane l owns chunks l and l + 32.  Put 2^24 in chunk 0 and
    # 1.0 in chunk 32 (same lane, added after) -> lost; 1.0 in chunk 1 (lane 1,
    # joined by the butterfly at offset 1 as 2^24 + 1) -> lost as well.
    v = np.zeros((1, 512), dtype=F32)
    v[0, 0] = 2.0 ** 24
    v[0, 32 * 8] = 1.0
    v[0, 1 * 8] = 1.0
    assert S.canonical_sum(v)[0] == F32(2.0 ** 24)
    # 1.0 in chunks 1 and 3 (lanes 1 and 3): the butterfly adds lane 1 + lane 3 first
    # (offset 2) giving 2.0, which survives the final add to 2^24.
    v[0, 32 * 8] = 0.0
    v[0, 3 * 8] = 1.0
    assert S.canonical_sum(v)[0] == F32(2.0 ** 24 + 2)


@pytest.mark.parametrize("D", [8, 64, 128, 264, 1024, 5120])
def test_canonical_sum_within_fp32_error_bound_of_exact(D):
    g = np.random.default_rng(D)
    v = np.abs(g.standard_normal((16, D))).astype(F32)
    got = S.canonical_sum(v).astype(np.float64)
    C = D // 8
    depth = 7 + (C + 31) // 32 + 5           # adds on the longest path
    for r in range(16):
        exact = math.fsum(float(t) for t in v[r])
        assert abs(got[r] - exact) <= depth * 2.0 ** -24 * exact * 1.0001


def test_drift_zero_when_input_equals_cache():
    q, s = G.random_cache(12, 64, seed=1)
    x = (q.astype(F32) * s[:, None]).astype(F32)
    assert (S.drift(x, q, s) == 0).all()


def test_drift_is_relative_l1_change():
    q, s = G.random_cache(10, 128, seed=2)
    x = G.random_rows(10, 128, seed=3)
    d = S.drift(x, q, s, xi=1e-6).astype(np.float64)
    c = q.astype(np.float64) * s[:, None].astype(np.float64)
    ref = np.abs(x - c).sum(1) / (np.abs(c).sum(1) + 1e-6)
    assert np.allclose(d, ref, rtol=1e-5)


def test_drift_of_zero_cache_is_l1_over_xi():
    x = np.zeros((2, 16), dtype=F32)
    x[0, 3] = -2.0
    q = np.zeros((2, 16), dtype=np.int8)
    s = np.zeros(2, dtype=F32)
    d = S.drift(x, q, s, xi=1e-6)
    assert d[0] == F32(2.0) / F32(1e-6) and d[1] == 0


@pytest.mark.parametrize("num,den,NT,K", [(1, 4, 256, 64), (1, 5, 7800, 1560), (1, 5, 32760, 6552),
                                         (1, 20, 63960, 3198), (1, 10, 63960, 6396),
                                         (1, 2, 63960, 31980), (1, 1, 63960, 63960),
                                         (0, 1, 100, 0), (1, 3, 7, 3), (2, 3, 7, 5)])
def test_refresh_budget_integer_ceiling(num, den, NT, K):
    assert S.refresh_budget(NT, num, den) == K


def _dominates(score, i, j):
    return score[i] > score[j] or (score[i] == score[j] and i < j)


@pytest.mark.parametrize("seed", range(8))
def test_top_k_equals_brute_force_over_all_subsets(seed):
    g = np.random.default_rng(seed)
    NT = int(g.integers(1, 11))
    # few distinct values so that ties are common
    score = g.integers(0, 4, size=NT).astype(F32) * F32(0.25)
    for K in range(NT + 1):
        winners = [set(c) for c in itertools.combinations(range(NT), K)
                   if all(_dominates(score, i, j) for i in c for j in range(NT) if j not in c)]
        assert len(winners) == 1
        assert list(S.top_k(score, K)) == sorted(winners[0])


def test_top_k_against_full_sort_and_extremes():
    g = np.random.default_rng(5)
    score = g.random(20000).astype(F32)
    score[::7] = score[3]                     # plant ties
    K = 4000
    ranked = sorted(range(20000), key=lambda i: (-float(score[i]), i))
    assert list(S.top_k(score, K)) == sorted(ranked[:K])
    assert len(S.top_k(score, 0)) == 0
    assert list(S.top_k(score, 20000)) == list(range(20000))


def test_segment_mode_fills_whole_loudest_segments():
    T, N = 6, 10
    e = np.array([1.0, 5.0, 3.0, 6.0, 0.5, 2.0], dtype=F32)
    x = np.zeros((T * N, 8), dtype=F32)
    q = np.zeros((T * N, 8), dtype=np.int8)
    s = np.zeros(T * N, dtype=F32)
    idx, _ = S.select(x, q, s, e, T, N, 1, 4, mode=S.MODE_SEGMENT)   # K = 15
    # segment 3 (all 10 tokens) then the first 5 tokens of segment 1
    assert list(idx) == list(range(10, 15)) + list(range(30, 40))


def test_energy_weight_breaks_equal_drift():
    T, N, D = 3, 4, 8
    q = np.zeros((T * N, D), dtype=np.int8)
    s = np.zeros(T * N, dtype=F32)
    x = np.ones((T * N, D), dtype=F32)        # identical drift for every token
    e = np.array([1.0, 3.0, 2.0], dtype=F32)
    idx, sc = S.select(x, q, s, e, T, N, 1, 3)  # K = 4 -> all of segment 1
    assert list(idx) == [4, 5, 6, 7]
    assert sc[4] > sc[8] > sc[0]


def test_ratio_one_selects_all_ratio_zero_none():
    q, s = G.random_cache(30, 16, seed=4)
    x = G.random_rows(30, 16, seed=5)
    e = G.random_energy(3, seed=6)
    assert list(S.select(x, q, s, e, 3, 10, 1, 1)[0]) == list(range(30))
    assert len(S.select(x, q, s, e, 3, 10, 0, 1)[0]) == 0


# ---- ablation selections (Sec. 4, Table 2: Uniform, Random) ----------------
@pytest.mark.parametrize("NT,K", [(256, 64), (32760, 6552), (7, 3), (10, 10), (10, 1), (5, 0)])
def test_uniform_selection_spacing(NT, K):
    idx = S.uniform(NT, K)
    assert len(idx) == K and idx.dtype == np.int32
    if K:
        assert idx[0] == 0 and np.all(np.diff(idx) > 0) and idx[-1] < NT
        gaps = np.diff(np.append(idx, NT))
        assert set(gaps.tolist()) <= {NT // K, -(-NT // K)}
        # every window of ceil(NT/K) consecutive tokens holds at least one selected token
        w = -(-NT // K)
        hit = np.zeros(NT + w, dtype=int)
        hit[idx] = 1
        assert min(hit[i:i + w].sum() for i in range(NT - w + 1)) >= 1


def test_random_subset_is_top_keys_and_uniform_in_frequency():
    g = np.random.default_rng(0)
    keys = g.random(12).astype(np.float32)
    K = 5
    # brute force: the subset of size K with the largest key sum is the top K
    import itertools
    best = max(itertools.combinations(range(12), K), key=lambda c: keys[list(c)].sum())
    assert S.random_subset(keys, K).tolist() == sorted(best)
    # equal keys: the lowest indices
    assert S.random_subset(np.zeros(9, dtype=np.float32), 4).tolist() == [0, 1, 2, 3]
    # with fresh uniform keys every token is picked with frequency K / NT
    NT, trials = 40, 4000
    cnt = np.zeros(NT)
    for _ in range(trials):
        cnt[S.random_subset(g.random(NT).astype(np.float32), 10)] += 1
    f = cnt / trials
    assert np.abs(f - 10 / NT).max() < 0.04
