"""Seeded synthetic inputs shared by the oracle and the CUDA path.

Nothing here computes any step of the method: this module only draws random
numbers, shapes them into the paper's workloads and rounds them to bf16 once,
so that both sides start from identical bytes.  Floating-point tensors come
back as float32 numpy arrays whose values are exactly representable in bf16
(the GPU side converts them with an exact cast).

Recipe (stated once, used everywhere):
  * generator: numpy PCG64; weights seed [0, layer], latents seed 1, audio
    seed 2, condition projection seed 3, per-step perturbation seed 100 + t;
  * weights and biases N(0, 0.02), rounded to bf16;
  * latents N(0, 1) rounded to bf16; step t input = bf16(x0 + sum_{s<=t} eps_s)
    with eps_s ~ N(0, 0.05^2) (a stand-in for the sampler, Sec. 3.1);
  * audio at 16 kHz in one of four profiles: speech-like (unit Gaussian noise
    amplitude-modulated at 3 Hz, two 150 ms silent gaps centred at L/3 and
    2L/3), silence, a 0.5-amplitude 440 Hz tone, 120 BPM beats (30 ms noise
    bursts, 10 ms exponential decay, on an N(0, 0.01^2) floor);
  * audio condition tokens: the audio cut into L_c equal chunks, each chunk
    projected to D by a fixed N(0, 1/sqrt(chunk)) matrix and scaled to unit
    RMS, rounded to bf16 (stand-in for the model's audio encoder).
"""
from __future__ import annotations

import numpy as np
import torch

from .configs import Workload

WEIGHT_NAMES = ("Wq", "bq", "Wk", "bk", "Wv", "bv", "Wo", "bo",
                "Wqc", "bqc", "Wkc", "bkc", "Wvc", "bvc", "Woc", "boc",
                "W1", "b1", "W2", "b2")


def rng(seed) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(seed))


def to_bf16_values(a: np.ndarray) -> np.ndarray:
    """Round float32 values to the nearest bf16 (ties to even); keep float32 storage."""
    t = torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32))
    return t.to(torch.bfloat16).to(torch.float32).numpy()


def weight_shapes(w: Workload) -> dict:
    D, F = w.D, w.F
    s = {}
    for p in ("q", "k", "v", "o", "qc", "kc", "vc", "oc"):
        s["W" + p] = (D, D)
        s["b" + p] = (D,)
    s["W1"], s["b1"] = (F, D), (F,)
    s["W2"], s["b2"] = (D, F), (D,)
    return s


def block_weights(w: Workload, layer: int = 0) -> dict:
    """nn.Linear-convention weights of one block: y = x @ W.T + b."""
    g = rng([0, layer])
    shapes = weight_shapes(w)
    out = {}
    for name in WEIGHT_NAMES:
        a = g.standard_normal(shapes[name], dtype=np.float32)
        a *= np.float32(0.02)
        out[name] = to_bf16_values(a)
    return out


def audio(w: Workload, profile: str | None = None) -> np.ndarray:
    profile = profile or w.profile
    L, sr = w.n_samples, w.sample_rate
    t = np.arange(L, dtype=np.float64) / sr
    g = rng(2)
    if profile == "silence":
        a = np.zeros(L)
    elif profile == "tone":
        a = 0.5 * np.sin(2.0 * np.pi * 440.0 * t)
    elif profile == "speech":
        a = g.standard_normal(L) * 0.5 * (1.0 - np.cos(2.0 * np.pi * 3.0 * t))
        half_gap = int(round(0.075 * sr))
        for c in (L // 3, (2 * L) // 3):
            a[max(0, c - half_gap):min(L, c + half_gap)] = 0.0
    elif profile == "beats":
        a = 0.01 * g.standard_normal(L)
        period, burst = int(round(0.5 * sr)), int(round(0.030 * sr))
        env = np.exp(-np.arange(burst) / (0.010 * sr))
        for start in range(0, L, period):
            n = min(burst, L - start)
            a[start:start + n] += g.standard_normal(n) * env[:n]
    else:
        raise ValueError(f"unknown audio profile {profile!r}")
    return a.astype(np.float32)


def cond_tokens(w: Workload, audio_samples: np.ndarray) -> np.ndarray:
    """[L_c, D] audio condition tokens (bf16 values)."""
    chunk = len(audio_samples) // w.Lc
    g = rng(3)
    proj = g.standard_normal((chunk, w.D)) / np.sqrt(chunk)
    chunks = audio_samples[:chunk * w.Lc].astype(np.float64).reshape(w.Lc, chunk)
    tok = chunks @ proj
    rms = np.sqrt(np.mean(tok * tok, axis=1, keepdims=True))
    tok = np.where(rms > 0, tok / np.where(rms > 0, rms, 1.0), 0.0)
    return to_bf16_values(tok.astype(np.float32))


def latents(w: Workload) -> np.ndarray:
    """x0: [NT, D] bf16 values."""
    return to_bf16_values(rng(1).standard_normal((w.NT, w.D), dtype=np.float32))


def latents_smooth(w: Workload, rho: float = 0.95) -> np.ndarray:
    """x0 with spatially adjacent tokens alike: along each row of W' tokens of
    a latent frame the rows follow an AR(1) chain, x_w = rho x_{w-1} +
    sqrt(1 - rho^2) e_w, e ~ N(0, 1) (seed 1), so neighbouring tokens have
    cosine similarity about rho, as in real video latents.  [NT, D] bf16 values."""
    e = rng(1).standard_normal((w.T * w.Hp, w.Wp, w.D), dtype=np.float32)
    c = np.float32(np.sqrt(1.0 - rho * rho))
    for k in range(1, w.Wp):
        e[:, k] = np.float32(rho) * e[:, k - 1] + c * e[:, k]
    return to_bf16_values(e.reshape(w.NT, w.D))


def step_input(w: Workload, x0: np.ndarray, t: int) -> np.ndarray:
    """Layer-0 input at step t: bf16(x0 + sum_{s=1..t} eps_s), eps_s ~ N(0, 0.05^2)."""
    acc = x0.astype(np.float32).copy()
    for s in range(1, t + 1):
        e = rng(100 + s).standard_normal(x0.shape, dtype=np.float32)
        e *= np.float32(0.05)
        acc += e
    return to_bf16_values(acc)


def step_inputs(w: Workload, x0: np.ndarray, steps: int):
    """The layer-0 inputs of steps 0 .. steps-1 in order: the same values as
    step_input(w, x0, t) for each t, drawn incrementally (one perturbation per
    step instead of t)."""
    acc = x0.astype(np.float32).copy()
    for t in range(steps):
        if t:
            e = rng(100 + t).standard_normal(x0.shape, dtype=np.float32)
            e *= np.float32(0.05)
            acc += e
        yield to_bf16_values(acc)


# ---- generic kernel-level inputs (for parity checks of single entry points) ----

def random_rows(n_rows: int, D: int, seed: int, scale: float = 1.0) -> np.ndarray:
    """[n_rows, D] bf16 values, N(0, scale^2)."""
    a = rng(seed).standard_normal((n_rows, D), dtype=np.float32) * np.float32(scale)
    return to_bf16_values(a)


def random_cache(n_rows: int, D: int, seed: int, zero_rows: int = 0):
    """An int8 per-token cache: q in [-127, 127], scales in [1e-3, 5e-2).

    The first `zero_rows` rows are all-zero with scale 0 (the state a zero row
    quantises to)."""
    g = rng(seed)
    q = g.integers(-127, 128, size=(n_rows, D), dtype=np.int8)
    s = g.uniform(1e-3, 5e-2, size=n_rows).astype(np.float32)
    q[:zero_rows] = 0
    s[:zero_rows] = 0.0
    return q, s


def random_energy(T: int, seed: int, distinct: bool = True) -> np.ndarray:
    """Per-segment energies (float32, positive)."""
    g = rng(seed)
    if distinct:
        e = g.permutation(T).astype(np.float32) + np.float32(1.0)
        return (e * np.float32(0.37)).astype(np.float32)
    return g.uniform(0.1, 3.0, size=T).astype(np.float32)


def step_output_pair(n: int, seed: int, change: float = 0.05, bf16: bool = True):
    """Two flat length-n outputs of consecutive steps: h_prev ~ N(0, 1) and
    h_cur = h_prev + N(0, change^2), both rounded to bf16 values when bf16."""
    g = rng(seed)
    a = g.standard_normal(n, dtype=np.float32)
    b = a + g.standard_normal(n, dtype=np.float32) * np.float32(change)
    if bf16:
        return to_bf16_values(a), to_bf16_values(b)
    return a, b


def correlated_rows(n: int, D: int, seed: int, rho: float = 0.95) -> np.ndarray:
    """[n, D] bf16 values; consecutive rows follow an AR(1) chain,
    x_i = rho x_{i-1} + sqrt(1 - rho^2) e_i with e ~ N(0, 1), so neighbouring
    rows have cosine similarity about rho (like spatially adjacent latents)."""
    g = rng(seed)
    e = g.standard_normal((n, D), dtype=np.float32)
    x = np.empty_like(e)
    if n:
        x[0] = e[0]
    c = np.float32(np.sqrt(1.0 - rho * rho))
    for i in range(1, n):
        x[i] = np.float32(rho) * x[i - 1] + c * e[i]
    return to_bf16_values(x)
