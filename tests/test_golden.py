"""The oracle against the hand-worked fixtures in tests/golden/."""
import json
import os

import numpy as np

from oracle import cache as C
from oracle import energy as E
from oracle import select as S

GOLD = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "hand_worked.json")))


def test_quant_half_even():
    g = GOLD["quant_half_even"]
    q, s, _ = C.quantize_rows(np.array([g["v"]], dtype=np.float32))
    assert list(q[0]) == g["q"] and s[0] == g["s"]


def test_dequant_bf16_ties():
    g = GOLD["dequant_bf16_ties"]
    out = C.dequantize_rows(np.array([g["q"]], dtype=np.int8), np.array([g["s"]], dtype=np.float32))
    assert list(out[0]) == g["out"]


def test_drift_order_within_chunk():
    for v, want in GOLD["drift_order_within_chunk"]["cases"]:
        assert S.canonical_sum(np.array([v], dtype=np.float32))[0] == np.float32(want)


def test_refresh_budget():
    for NT, num, den, K in GOLD["refresh_budget"]["cases"]:
        assert S.refresh_budget(NT, num, den) == K


def test_hann_cosine_at_bin():
    g = GOLD["hann_cosine_at_bin"]
    N, k0 = g["N"], g["k0"]
    n = np.arange(N)
    P = E.dft_power((np.cos(2 * np.pi * k0 * n / N) * E.hann_periodic(N))[None], N)[0]
    assert abs(P[k0] - g["P_k0"]) < 1e-9 and abs(P[k0 + 1] - g["P_neighbour"]) < 1e-9


def test_ref_cache_scan():
    from oracle import refcache as R
    g = GOLD["ref_cache_scan"]
    v = np.array(g["rows"], dtype=np.float32)
    c = R.RefCache(len(v), v.shape[1], g["R_cap"], g["seg_len"], g["tau"])
    rows = np.arange(len(v))
    assert c.scan(rows, v).tolist() == g["src"]
    c.write(rows, v)
    assert c.ref.tolist() == g["ref"] and c.refcount.tolist() == g["refcount"]
