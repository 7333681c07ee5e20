"""Per-token drift score and energy-weighted refresh selection.

TEST INFRASTRUCTURE ONLY (see the package header).

Drift (Eq. 1, Sec. 3.1; used per token in Sec. 3.3).  Eq. 1 is a step-level
relative L1 change.  Reading: applied per token between the current layer input
x_i and that token's cached feature c_i (what reuse would return), with
c_i reconstructed from the int8 cache as in Sec. 3.4:
    d_i = sum_j |x_ij - c_ij| / (sum_j |c_ij| + xi),   c_ij = float(q_ij) * s_i.
xi is "a small constant" in the paper; xi = 1e-6.

Both sums are fp32 in a fixed canonical order, so that results are bit-exact
and reproducible on any hardware:
  * the row is cut into chunks of 8 consecutive elements, chunk c holds
    elements 8c .. 8c+7; lane l (0..31) owns chunks l, l+32, l+64, ...;
  * a chunk is summed left to right; each lane adds its chunk sums in chunk
    order to an accumulator that starts at 0;
  * the 32 lane accumulators are combined by a butterfly: for o = 16, 8, 4, 2, 1
    every lane adds the accumulator of lane (l xor o); lane 0's value is the sum.
Every operation is one IEEE fp32 round-to-nearest add, multiply or divide.

Selection (Sec. 3.3, "Cross-modal Saliency Anchors" and "Energy-Guided
Step-Latent Cache Scheduling").  The paper selects high-energy segments by
top-k, builds the latent mask [B, T, N, 1] flattened to [B, T*N, 1] and sets
the per-step budget k_t = ceil(N r_t).  Reading: one global budget
K = ceil(r NT) in integer arithmetic; token i belongs to segment floor(i / N);
score_i = w_{floor(i/N)} * d_i (fp32); the K tokens with the largest key
(score descending, index ascending) are active, returned as an ascending index
list (the compact form of the mask).  Mode SEGMENT is the paper-literal anchor:
d_i = 1 and lam = 0, so whole high-energy segments fill the budget in index order.

The ablation selections of Sec. 4 (Uniform, Random) take neither energy nor
drift: `uniform` spaces K tokens evenly, `random_subset` takes the top K of
keys the caller draws.

Pins: brute force over all subsets on tiny inputs, a full sort, r = 0 / r = 1,
x == c gives 0, the canonical order on hand-built cases where order matters,
an fp32 error bound against the exact sum; uniform spacing by counting,
random subsets by the brute-force top-K and by frequency.
"""
from __future__ import annotations

import numpy as np

from .energy import segment_weights

MODE_ENERGY_DRIFT = 0
MODE_SEGMENT = 1
MODE_DRIFT_ONLY = 2

CHUNK = 8
LANES = 32


def canonical_sum(v: np.ndarray) -> np.ndarray:
    """fp32 row sums of v [R, D] (D % 8 == 0) in the canonical order above."""
    v = np.asarray(v, dtype=np.float32)
    R, D = v.shape
    if D % CHUNK:
        raise ValueError("D must be a multiple of 8")
    C = D // CHUNK
    ch = v.reshape(R, C, CHUNK)
    cs = ch[:, :, 0].copy()
    for e in range(1, CHUNK):
        cs = (cs + ch[:, :, e]).astype(np.float32)
    acc = np.zeros((R, LANES), dtype=np.float32)
    for it in range(0, C, LANES):
        n = min(LANES, C - it)
        acc[:, :n] = (acc[:, :n] + cs[:, it:it + n]).astype(np.float32)
    lanes = np.arange(LANES)
    for o in (16, 8, 4, 2, 1):
        acc = (acc + acc[:, lanes ^ o]).astype(np.float32)
    return acc[:, 0].copy()


def dequant_f32(q: np.ndarray, s: np.ndarray) -> np.ndarray:
    """c_ij = float(q_ij) * s_i, one fp32 multiply."""
    return (np.asarray(q).astype(np.float32) * np.asarray(s, dtype=np.float32)[:, None]).astype(np.float32)


def drift(x: np.ndarray, q: np.ndarray, s: np.ndarray, xi: float = 1e-6) -> np.ndarray:
    """d_i of Eq. 1 per token, fp32 [NT]."""
    return drift_from(x, dequant_f32(q, s), xi)


def drift_from(x: np.ndarray, c: np.ndarray, xi: float = 1e-6) -> np.ndarray:
    """d_i of Eq. 1 against an fp32 reconstruction c of any cache form."""
    x = np.asarray(x, dtype=np.float32)
    c = np.asarray(c, dtype=np.float32)
    num = canonical_sum(np.abs((x - c).astype(np.float32)))
    den = canonical_sum(np.abs(c))
    return (num / (den + np.float32(xi)).astype(np.float32)).astype(np.float32)


def refresh_budget(NT: int, ratio_num: int, ratio_den: int) -> int:
    """K = ceil(ratio_num * NT / ratio_den), integers only."""
    if ratio_den <= 0 or ratio_num < 0 or ratio_num > ratio_den:
        raise ValueError("ratio must lie in [0, 1]")
    return (ratio_num * NT + ratio_den - 1) // ratio_den


def scores(x, q, s, seg_energy, T: int, N: int, lam: float = 0.1, xi: float = 1e-6,
           mode: int = MODE_ENERGY_DRIFT) -> np.ndarray:
    """score_i = w_{floor(i/N)} * d_i in fp32."""
    return scores_from(x, None if mode == MODE_SEGMENT else dequant_f32(q, s), seg_energy, T, N,
                       lam, xi, mode)


def scores_from(x, c, seg_energy, T: int, N: int, lam: float = 0.1, xi: float = 1e-6,
                mode: int = MODE_ENERGY_DRIFT) -> np.ndarray:
    """scores against an fp32 reconstruction c of any cache form."""
    NT = T * N
    if mode == MODE_SEGMENT:
        w = segment_weights(seg_energy, 0.0)
        d = np.ones(NT, dtype=np.float32)
    elif mode == MODE_DRIFT_ONLY:
        w = np.ones(T, dtype=np.float32)
        d = drift_from(x, c, xi)
    else:
        w = segment_weights(seg_energy, lam)
        d = drift_from(x, c, xi)
    wt = np.repeat(w, N)
    return (wt * d).astype(np.float32)


def top_k(score: np.ndarray, K: int) -> np.ndarray:
    """Ascending int32 indices of the K largest (score desc, index asc)."""
    score = np.asarray(score, dtype=np.float32)
    NT = score.shape[0]
    order = np.lexsort((np.arange(NT), -score.astype(np.float64)))
    return np.sort(order[:K]).astype(np.int32)


def uniform(NT: int, K: int) -> np.ndarray:
    """Uniform selection (the "Uniform" ablation of Sec. 4, Table 2): K tokens
    evenly spaced over the token order, idx_j = floor(j NT / K), integers only."""
    if K <= 0:
        return np.zeros(0, dtype=np.int32)
    return (np.arange(K, dtype=np.int64) * NT // K).astype(np.int32)


def random_subset(keys: np.ndarray, K: int) -> np.ndarray:
    """Random selection (the "Random" ablation of Sec. 4, Table 2): the K tokens
    with the largest caller-drawn keys (key desc, index asc); with keys drawn
    independently and uniformly this is a uniformly random K-subset."""
    return top_k(np.asarray(keys, dtype=np.float32), K)


def select(x, q, s, seg_energy, T: int, N: int, ratio_num: int, ratio_den: int,
           lam: float = 0.1, xi: float = 1e-6, mode: int = MODE_ENERGY_DRIFT):
    """Returns (idx int32[K] ascending, scores fp32[NT])."""
    sc = scores(x, q, s, seg_energy, T, N, lam, xi, mode)
    K = refresh_budget(T * N, ratio_num, ratio_den)
    return top_k(sc, K), sc
