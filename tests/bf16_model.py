"""An ideal bf16 tensor-core block: the oracle's block with only the unavoidable
bf16 roundings added.

A bf16 tensor-core path must hold the operands of its contractions in bf16:
the layer-norm outputs, Q, K and V, the softmax probabilities P, the attention
outputs, the FFN hidden layer, and the block output (the workload's storage
type).  This model rounds exactly those values to bf16 (round to nearest
even) and computes everything else in fp64, with the oracle's own layer norm,
GELU and linear maps.  Its error against the fp64 oracle is the floor that
any bf16 path reaches, so the GPU's element-wise error is compared against
this model's element-wise error on the same rows.

Test helper only: it builds on `oracle.block` and is used by the tests.
"""
from __future__ import annotations

import numpy as np
import torch

import oracle

B = oracle.block


def bf(a) -> np.ndarray:
    """Values rounded to bf16 (ties to even), returned as fp64."""
    t = torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(torch.bfloat16)
    return t.to(torch.float32).numpy().astype(np.float64)


def mha_bf16_p(Q, K, V, H: int) -> np.ndarray:
    """Attention with P rounded to bf16 before P V; the row sum stays exact."""
    M, D = Q.shape
    d = D // H
    out = np.empty((M, D))
    for h in range(H):
        sl = slice(h * d, (h + 1) * d)
        S = Q[:, sl] @ K[:, sl].T / np.sqrt(d)
        P = np.exp(S - S.max(axis=1, keepdims=True))
        out[:, sl] = (bf(P) @ V[:, sl]) / P.sum(axis=1, keepdims=True)
    return out


def self_kv(x, W, fp32: bool = False):
    """bf16 K and V over every token from the bf16 layer norm of x.  With fp32
    the product of the (exactly representable) bf16 operands is accumulated in
    fp32, which is far below the bf16 rounding of the result and much faster at
    the full sizes."""
    n1 = bf(B.layer_norm(x))
    if fp32:
        n1f = n1.astype(np.float32)
        K = n1f @ W["Wk"].astype(np.float32).T + W["bk"].astype(np.float32)
        V = n1f @ W["Wv"].astype(np.float32).T + W["bv"].astype(np.float32)
        return bf(K), bf(V)
    return bf(B.linear(n1, W["Wk"], W["bk"])), bf(B.linear(n1, W["Wv"], W["bv"]))


def cross_kv(cond, W):
    return bf(B.linear(cond, W["Wkc"], W["bkc"])), bf(B.linear(cond, W["Wvc"], W["bvc"]))


def active_rows(x, rows, W, H: int, Kv, Vv, Kc, Vc) -> np.ndarray:
    """y_act of `rows` given the model's bf16 K/V (self_kv, cross_kv)."""
    x = np.asarray(x, dtype=np.float64)
    xa = x[np.asarray(rows)]
    Q = bf(B.linear(bf(B.layer_norm(xa)), W["Wq"], W["bq"]))
    h1 = xa + B.linear(bf(mha_bf16_p(Q, Kv, Vv, H)), W["Wo"], W["bo"])
    Qc = bf(B.linear(bf(B.layer_norm(h1)), W["Wqc"], W["bqc"]))
    h2 = h1 + B.linear(bf(mha_bf16_p(Qc, Kc, Vc, H)), W["Woc"], W["boc"])
    u = bf(B.gelu_tanh(B.linear(bf(B.layer_norm(h2)), W["W1"], W["b1"])))
    return bf(h2 + B.linear(u, W["W2"], W["b2"]))


def block_active(x, rows, W, cond, H: int) -> np.ndarray:
    Kv, Vv = self_kv(x, W)
    Kc, Vc = cross_kv(cond, W)
    return active_rows(x, rows, W, H, Kv, Vv, Kc, Vc)


def elementwise_rel(g, o) -> float:
    """max over elements of |g - o| / max(|o|, 0.1 rms(o_row)): the element-wise
    reading of "max relative error" with a floor at a tenth of the row's rms."""
    g = np.asarray(g, dtype=np.float64)
    o = np.asarray(o, dtype=np.float64)
    den = np.maximum(np.abs(o), 0.1 * np.sqrt((o * o).mean(axis=-1, keepdims=True)))
    return float((np.abs(g - o) / den).max())


def normwise_rel(g, o):
    """(max over rows of max_j|g - o| / max_j|o|, sum|g - o| / sum|o|)."""
    g = np.asarray(g, dtype=np.float64)
    o = np.asarray(o, dtype=np.float64)
    nw = np.abs(g - o).max(axis=-1) / np.abs(o).max(axis=-1)
    return float(nw.max()), float(np.abs(g - o).sum() / np.abs(o).sum())
