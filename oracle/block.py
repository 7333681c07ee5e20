"""The DiT block on active latents (Sec. 3.3, "Fine-grained latent-level caching").

TEST INFRASTRUCTURE ONLY (see the package header).

The paper fixes what is computed for whom: queries only for the active
latents, keys and values from the complete latent set, attention on
(Q', K, V), the FFN only on active latents, and a mask fusion with the cache
after the attention and again after the FFN residual.  It does not give the
block's internals.  Reading: a plain pre-LN DiT block with self-attention over
the video latent tokens, cross-attention to the audio condition tokens and a
GELU FFN (the denoiser f_theta(x_t, t, y) of Sec. 3.1 reduced to one block):
  LN(v)  = (v - mean) / sqrt(var + 1e-6), biased variance, no affine;
  n1     = LN(x) for all NT rows;  K = n1 Wk^T + bk,  V = n1 Wv^T + bv  (all rows);
  Q'     = n1[idx] Wq^T + bq       (active rows);
  h1     = x[idx] + MHA(Q', K, V) Wo^T + bo;
  h2     = h1 + MHA(LN(h1) Wqc^T + bqc, Kc, Vc) Woc^T + boc,
           Kc = cond Wkc^T + bkc, Vc = cond Wvc^T + bvc;
  y_act  = h2 + GELU_tanh(LN(h2) W1^T + b1) W2^T + b2,
  MHA per head h of width d: softmax(Q_h K_h^T / sqrt(d)) V_h;
  GELU_tanh(u) = u/2 (1 + tanh(sqrt(2/pi) (u + 0.044715 u^3))) (Hendrycks & Gimpel).
With one block-output cache the two fusions collapse into one merge (the
inactive rows skip every position-wise op, so the first fusion only feeds the
active rows): y[i] = y_act[j] if i = idx[j], else the reconstructed cache.
Everything here is fp64 on the bf16-valued inputs.

Pins: layer norm, GELU and attention against torch's fp64 routines, attention
with one key and with identical keys, key permutation invariance, the whole
block against a torch.nn composition (MultiheadAttention, LayerNorm, GELU) in
fp64, and active rows equal to the uncached block's rows.
"""
from __future__ import annotations

import numpy as np

LN_EPS = 1e-6


def layer_norm(v: np.ndarray, eps: float = LN_EPS) -> np.ndarray:
    v = np.asarray(v, dtype=np.float64)
    mu = v.mean(axis=-1, keepdims=True)
    var = ((v - mu) ** 2).mean(axis=-1, keepdims=True)
    return (v - mu) / np.sqrt(var + eps)


def gelu_tanh(u: np.ndarray) -> np.ndarray:
    u = np.asarray(u, dtype=np.float64)
    return 0.5 * u * (1.0 + np.tanh(np.sqrt(2.0 / np.pi) * (u + 0.044715 * u ** 3)))


def linear(v: np.ndarray, W: np.ndarray, b: np.ndarray) -> np.ndarray:
    return np.asarray(v, dtype=np.float64) @ np.asarray(W, dtype=np.float64).T + np.asarray(b, dtype=np.float64)


def mha(Q: np.ndarray, K: np.ndarray, V: np.ndarray, H: int) -> np.ndarray:
    """softmax(Q_h K_h^T / sqrt(d)) V_h per head; Q [M, H d], K/V [L, H d]."""
    M, D = Q.shape
    d = D // H
    out = np.empty((M, D))
    for h in range(H):
        sl = slice(h * d, (h + 1) * d)
        S = Q[:, sl] @ K[:, sl].T / np.sqrt(d)
        S = S - S.max(axis=1, keepdims=True)
        P = np.exp(S)
        P /= P.sum(axis=1, keepdims=True)
        out[:, sl] = P @ V[:, sl]
    return out


def self_kv(x: np.ndarray, W: dict):
    """K and V for every latent token (Q', K, V of Sec. 3.3: K/V from all latents)."""
    n1 = layer_norm(x)
    return linear(n1, W["Wk"], W["bk"]), linear(n1, W["Wv"], W["bv"])


def cross_kv(cond: np.ndarray, W: dict):
    return linear(cond, W["Wkc"], W["bkc"]), linear(cond, W["Wvc"], W["bvc"])


def active_rows(x: np.ndarray, idx: np.ndarray, W: dict, H: int, Kv, Vv, Kc, Vc) -> np.ndarray:
    """y_act [len(idx), D] for the active tokens, given all-token K/V."""
    x = np.asarray(x, dtype=np.float64)
    xa = x[np.asarray(idx)]
    Qp = linear(layer_norm(xa), W["Wq"], W["bq"])
    h1 = xa + linear(mha(Qp, Kv, Vv, H), W["Wo"], W["bo"])
    Qc = linear(layer_norm(h1), W["Wqc"], W["bqc"])
    h2 = h1 + linear(mha(Qc, Kc, Vc, H), W["Woc"], W["boc"])
    u = gelu_tanh(linear(layer_norm(h2), W["W1"], W["b1"]))
    return h2 + linear(u, W["W2"], W["b2"])


def block_active(x, idx, W: dict, cond, H: int) -> np.ndarray:
    Kv, Vv = self_kv(x, W)
    Kc, Vc = cross_kv(cond, W)
    return active_rows(x, idx, W, H, Kv, Vv, Kc, Vc)


def uncached_block(x, W: dict, cond, H: int) -> np.ndarray:
    """The plain block on every token, no cache (the r = 1 reference)."""
    x = np.asarray(x, dtype=np.float64)
    n1 = layer_norm(x)
    Q = linear(n1, W["Wq"], W["bq"])
    Kv = linear(n1, W["Wk"], W["bk"])
    Vv = linear(n1, W["Wv"], W["bv"])
    h1 = x + linear(mha(Q, Kv, Vv, H), W["Wo"], W["bo"])
    Kc, Vc = cross_kv(cond, W)
    h2 = h1 + linear(mha(linear(layer_norm(h1), W["Wqc"], W["bqc"]), Kc, Vc, H), W["Woc"], W["boc"])
    return h2 + linear(gelu_tanh(linear(layer_norm(h2), W["W1"], W["b1"])), W["W2"], W["b2"])


def merge(y_act: np.ndarray, idx: np.ndarray, cached: np.ndarray) -> np.ndarray:
    """x_out = m * x_new + (1 - m) * x_cached with m the active mask (Sec. 3.3)."""
    out = np.array(cached, dtype=np.float64, copy=True)
    out[np.asarray(idx)] = y_act
    return out
