"""int8 per-token cache: quantisation and reconstruction (Sec. 3.4).

TEST INFRASTRUCTURE ONLY (see the package header).

The paper stores cache entries as int8 (residuals against a reference in its
full design; its ablation also runs a plain int8 cache) and converts the
reconstruction back to the compute precision.  It gives no granularity,
rounding or clamp.  Readings, fp32 arithmetic in this order:
  quantise a row v (fp32 values of the bf16 storage):
    a = max_j |v_j|;  a == 0 -> s = 0, q = 0;
    else s = a / 127, inv = 127 / a, q_j = clamp(round_half_even(v_j * inv), -127, 127);
    a non-finite -> the row is flagged (NONFINITE) and written as q = 0, s = a;
  reconstruct: c_j = float(q_j) * s (one fp32 multiply), then bf16 round to
    nearest even ("converted back to the original computation precision").

Pins: |v - q s| <= s (1/2 + 2^-14) (the rounding bound plus the three fp32
roundings of s, inv and v * inv), a zero row, sign symmetry, the largest
element maps to +-127, hand-worked ties.
"""
from __future__ import annotations

import numpy as np


def round_bf16(a: np.ndarray) -> np.ndarray:
    """Round fp32 values to bf16, nearest even; returns fp32 storage."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    u = a.view(np.uint32).astype(np.uint64)
    lsb = (u >> np.uint64(16)) & np.uint64(1)
    r = ((u + np.uint64(0x7FFF) + lsb) >> np.uint64(16)) << np.uint64(16)
    out = r.astype(np.uint32).view(np.float32).copy()
    nan = np.isnan(a)
    out[nan] = np.float32(np.nan)
    return out


def quantize_rows(v: np.ndarray):
    """Returns (q int8 [R, D], s fp32 [R], nonfinite bool [R])."""
    v = np.asarray(v, dtype=np.float32)
    R, D = v.shape
    a = np.abs(v).max(axis=1) if D else np.zeros(R, dtype=np.float32)
    a = a.astype(np.float32)
    q = np.zeros((R, D), dtype=np.int8)
    s = np.zeros(R, dtype=np.float32)
    bad = ~np.isfinite(a)
    ok = (a > 0) & ~bad
    if ok.any():
        aa = a[ok]
        s[ok] = (aa / np.float32(127.0)).astype(np.float32)
        inv = (np.float32(127.0) / aa).astype(np.float32)
        t = (v[ok] * inv[:, None]).astype(np.float32)
        q[ok] = np.clip(np.rint(t), -127, 127).astype(np.int8)
    s[bad] = a[bad]
    return q, s, bad


def dequantize_rows(q: np.ndarray, s: np.ndarray) -> np.ndarray:
    """bf16(float(q) * s), fp32 storage [R, D]."""
    c = (np.asarray(q).astype(np.float32) * np.asarray(s, dtype=np.float32)[:, None]).astype(np.float32)
    return round_bf16(c)


def quant_scatter(src: np.ndarray, rows, q_cache: np.ndarray, s_cache: np.ndarray):
    """q_cache[rows[j]] = Q(src[j]) in place (rows None = identity)."""
    q, s, bad = quantize_rows(src)
    r = np.arange(src.shape[0]) if rows is None else np.asarray(rows)
    q_cache[r] = q
    s_cache[r] = s
    return bool(bad.any())


def dequant_gather(q_cache: np.ndarray, s_cache: np.ndarray, rows=None) -> np.ndarray:
    """dst[j] = bf16(q[rows[j]] * s[rows[j]]) (rows None = all)."""
    if rows is None:
        return dequantize_rows(q_cache, s_cache)
    r = np.asarray(rows)
    return dequantize_rows(q_cache[r], s_cache[r])
