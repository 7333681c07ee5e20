"""Why block outputs are compared with a per-token (normwise) max relative error.

The stated bar for bf16 block outputs against the fp32/fp64 oracle is 2e-2 max
relative and 5e-3 mean relative, without a denominator.  This test runs the
oracle's block twice on the CPU: once in fp64, once with every value that a
bf16 tensor-core path must hold in bf16 rounded to bf16 (the GEMM and attention
operands: LN outputs, Q/K/V, P, the attention output, the FFN hidden layer, and
the output) and nothing else.  Even this ideal bf16 path exceeds 2e-2 under an
elementwise reading with a 0.1 rms floor at D = 1024, while its per-token
normwise error max_j|g-o| / max_j|o| and its mean relative error stay far below
the bar.  The GPU tests therefore use the normwise reading for "max relative".
"""
import numpy as np
import torch

import oracle
from synth import generate as G, small

B = oracle.block


def bf(a):
    t = torch.from_numpy(np.asarray(a, np.float32)).to(torch.bfloat16)
    return t.to(torch.float32).numpy().astype(np.float64)


def mha_bf16_p(Q, K, V, H):
    M, D = Q.shape
    d = D // H
    out = np.empty((M, D))
    for h in range(H):
        sl = slice(h * d, (h + 1) * d)
        S = Q[:, sl] @ K[:, sl].T / np.sqrt(d)
        P = np.exp(S - S.max(axis=1, keepdims=True))
        out[:, sl] = (bf(P) @ V[:, sl]) / P.sum(axis=1, keepdims=True)
    return out


def ideal_bf16_block(x, idx, W, cond, H):
    n1 = bf(B.layer_norm(x))
    Kv, Vv = bf(B.linear(n1, W["Wk"], W["bk"])), bf(B.linear(n1, W["Wv"], W["bv"]))
    Q = bf(B.linear(n1[idx], W["Wq"], W["bq"]))
    h1 = x[idx] + B.linear(bf(mha_bf16_p(Q, Kv, Vv, H)), W["Wo"], W["bo"])
    Kc, Vc = bf(B.linear(cond, W["Wkc"], W["bkc"])), bf(B.linear(cond, W["Wvc"], W["bvc"]))
    Qc = bf(B.linear(bf(B.layer_norm(h1)), W["Wqc"], W["bqc"]))
    h2 = h1 + B.linear(bf(mha_bf16_p(Qc, Kc, Vc, H)), W["Woc"], W["boc"])
    u = bf(B.gelu_tanh(B.linear(bf(B.layer_norm(h2)), W["W1"], W["b1"])))
    return bf(h2 + B.linear(u, W["W2"], W["b2"]))


def test_elementwise_floor_reading_is_out_of_reach_for_bf16_operands():
    w = small(T=4, Hp=16, Wp=16, D=1024, H=16, d=64, F=4096, Lc=40, n_samples=16000)
    W = G.block_weights(w, 0)
    audio = G.audio(w)
    cond = G.cond_tokens(w, audio)
    x = G.latents(w).astype(np.float64)
    idx = np.sort(np.random.default_rng(0).choice(w.NT, 256, replace=False))
    ref = B.block_active(x, idx, W, cond, w.H)
    g = ideal_bf16_block(x, idx, W, cond, w.H)
    den = np.maximum(np.abs(ref), 0.1 * np.sqrt((ref ** 2).mean(axis=1, keepdims=True)))
    elementwise = (np.abs(g - ref) / den).max()
    normwise = (np.abs(g - ref).max(axis=1) / np.abs(ref).max(axis=1)).max()
    mean_rel = np.abs(g - ref).sum() / np.abs(ref).sum()
    assert elementwise > 2e-2          # the floored elementwise reading fails for any bf16 path
    assert normwise < 1e-2 and mean_rel < 5e-3
