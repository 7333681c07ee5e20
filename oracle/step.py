"""One cached layer step and the step loop (Sec. 3.3, "Energy-Guided Step-Latent Cache Scheduling").

TEST INFRASTRUCTURE ONLY (see the package header).

A cached layer step, in the paper's order: score and select the active
latents (energy-guided), run the block on them (Q' on active, K/V on all),
fuse with the reconstructed cache, write the active rows back into the int8
cache.  The paper keeps full computation in the early steps; the number of
such steps is not given.  Reading: step 0 is a full step (K = NT) that fills
every layer's cache; later steps use the fixed ratio r, or the adaptive r_t
of the paper (schedule.py) when a schedule is given.  Layer I/O is stored as bf16 (the
workload's storage type): the merged output is rounded to bf16 before it feeds
the next layer, and the cache quantises the bf16 value of y_act.

Pins: r = 1 equals the uncached block, r = 0 returns the reconstructed cache,
the step loop at r = 1 equals the uncached stack.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np

from . import block, cache, energy, select


@dataclass
class LayerResult:
    idx: np.ndarray          # int32 [K] ascending
    scores: np.ndarray       # fp32 [NT] (zeros on a full step)
    y_act: np.ndarray        # fp64 [K, D], the block output of the active rows
    y: np.ndarray            # fp64 [NT, D], merged output
    y_bf16: np.ndarray       # fp32 storage of bf16(y), the next layer's input
    q: np.ndarray            # int8 [NT, D], cache after the write
    s: np.ndarray            # fp32 [NT]
    nonfinite: bool


def cached_layer_step(x, q, s, seg_energy, W, cond, T, N, H, ratio_num, ratio_den,
                      lam=0.1, xi=1e-6, mode=select.MODE_ENERGY_DRIFT, full=False,
                      idx=None) -> LayerResult:
    NT = T * N
    if idx is not None:
        idx = np.asarray(idx, dtype=np.int32)
        sc = np.zeros(NT, dtype=np.float32)
    elif full:
        idx = np.arange(NT, dtype=np.int32)
        sc = np.zeros(NT, dtype=np.float32)
    else:
        idx, sc = select.select(x, q, s, seg_energy, T, N, ratio_num, ratio_den, lam, xi, mode)
    cached = cache.dequantize_rows(q, s)
    if len(idx):
        y_act = block.block_active(x, idx, W, cond, H)
    else:
        y_act = np.zeros((0, x.shape[1]))
    y = block.merge(y_act, idx, cached)
    q2, s2 = q.copy(), s.copy()
    bad = False
    if len(idx):
        bad = cache.quant_scatter(cache.round_bf16(y_act.astype(np.float32)), idx, q2, s2)
    y_bf16 = cache.round_bf16(y.astype(np.float32))
    return LayerResult(idx, sc, y_act, y, y_bf16, q2, s2, bad)


@dataclass
class CacheLayerResult:
    idx: np.ndarray          # int32 [K] ascending
    scores: np.ndarray       # fp32 [NT] (zeros on a full step)
    y_act: np.ndarray        # fp64 [K, D]
    y: np.ndarray            # fp64 [NT, D], merged output
    y_bf16: np.ndarray       # fp32 storage of bf16(y)
    cache: object            # the cache after the write (a copy)
    nonfinite: bool


def cached_layer_step_cache(x, c, seg_energy, W, cond, T, N, H, ratio_num, ratio_den,
                            lam=0.1, xi=1e-6, mode=select.MODE_ENERGY_DRIFT, full=False,
                            idx=None) -> CacheLayerResult:
    """The cached layer step with any cache form of refcache.py (Int8Cache,
    FullCache, RefCache): the drift is taken against the form's fp32
    reconstruction, inactive rows take its bf16 reconstruction, and the
    refreshed rows are written through the form's own write.  The input cache
    `c` is not modified."""
    NT = T * N
    if idx is not None:
        idx = np.asarray(idx, dtype=np.int32)
        sc = np.zeros(NT, dtype=np.float32)
    elif full:
        idx = np.arange(NT, dtype=np.int32)
        sc = np.zeros(NT, dtype=np.float32)
    else:
        rec = None if mode == select.MODE_SEGMENT else c.reconstruct_f32()
        sc = select.scores_from(x, rec, seg_energy, T, N, lam, xi, mode)
        idx = select.top_k(sc, select.refresh_budget(NT, ratio_num, ratio_den))
    cached = c.reconstruct_bf16()
    if len(idx):
        y_act = block.block_active(x, idx, W, cond, H)
    else:
        y_act = np.zeros((0, x.shape[1]))
    y = block.merge(y_act, idx, cached)
    c2 = c.copy()
    bad = False
    if len(idx):
        bad = c2.write(idx, cache.round_bf16(y_act.astype(np.float32)))
    return CacheLayerResult(idx, sc, y_act, y, cache.round_bf16(y.astype(np.float32)), c2, bad)


def generation(x_inputs, weights, cond, seg_energy, T, N, H, ratio_num, ratio_den,
               lam=0.1, xi=1e-6, mode=select.MODE_ENERGY_DRIFT, warmup_steps=1,
               record=None, rate=None):
    """Step loop over len(x_inputs) steps and len(weights) layers.

    x_inputs[t] is the layer-0 input at step t; layer l+1 takes layer l's merged
    output.  Steps < warmup_steps are full.  `record(t, l, x, q, s, result)` is
    called for every layer step with that step's inputs.  With `rate` (a
    schedule.Schedule) the cached steps take the adaptive budget of Sec. 3.3
    instead of ratio_num / ratio_den: every layer of step t refreshes
    K_t = rate.budget() tokens, and after each step rate.observe() gets the
    last layer's output of the step before and of this one.  Returns the final
    per-layer caches."""
    NT, D = x_inputs[0].shape
    L = len(weights)
    qs = [np.zeros((NT, D), dtype=np.int8) for _ in range(L)]
    ss = [np.zeros(NT, dtype=np.float32) for _ in range(L)]
    h_prev = None
    for t, x0 in enumerate(x_inputs):
        x = x0
        full = t < warmup_steps
        num, den = ratio_num, ratio_den
        if rate is not None and not full:
            num, den = rate.budget(), NT
        for l in range(L):
            r = cached_layer_step(x, qs[l], ss[l], seg_energy, weights[l], cond[l], T, N, H,
                                  num, den, lam, xi, mode, full=full)
            if record is not None:
                record(t, l, x, qs[l], ss[l], r)
            qs[l], ss[l] = r.q, r.s
            x = r.y_bf16
        if rate is not None:
            if h_prev is not None:
                rate.observe(h_prev, x)
            h_prev = x
    return qs, ss


def uncached_stack(x, weights, cond, H):
    """Every layer on every token, no cache, bf16 layer I/O."""
    for l in range(len(weights)):
        x = cache.round_bf16(block.uncached_block(x, weights[l], cond[l], H).astype(np.float32))
    return x


def audio_to_weights(audio, T, n_fft=512, hop=160, n_bands=8, lam=0.1):
    """energy (fp32 cast of the fp64 oracle value) and the per-segment weight."""
    band, e = energy.audio_energy(audio, T, n_fft, hop, n_bands)
    e32 = e.astype(np.float32)
    return band, e32, energy.segment_weights(e32, lam)
