"""Cache forms of Sec. 3.4 and of the quantisation ablation (Sec. 4, Table 2).

TEST INFRASTRUCTURE ONLY (see the package header).

Three forms of one layer's cache of NT token rows, all with the same interface
(reconstruct in fp32 for the drift score, reconstruct in bf16 for the merge,
write the refreshed rows):

  Int8Cache  the plain int8 per-token cache of cache.py ("Naive INT8").
  FullCache  the rows themselves in the compute precision (the "FP16" ablation;
             the compute precision here is bf16).
  RefCache   the paper's manager: a token is stored either as a reference (its
             row in full precision) or as an int8 residual against the current
             reference, chosen by cosine similarity against a threshold tau;
             references are reference-counted and released when no token
             refers to them any more.

RefCache readings (the paper gives the rule, not these details):
  * granularity: one token row of D values;
  * the running reference: the rows written in one call are scanned in
    ascending token order within scan segments of seg_len consecutive tokens
    (segment floor(i / seg_len); seg_len = W' makes a segment one spatial row
    of a latent frame, the "adjacent latents"); the first written row of a
    segment becomes a reference; a later row becomes the new reference when
    sim(x, r) <= tau, else it is stored as the residual x - r;
  * sim(x, r) = <x, r> / (sqrt(<x, x>) sqrt(<r, r>)) in fp32, the three sums in
    the canonical order of select.canonical_sum, products and the final sqrt,
    multiply and divide one IEEE fp32 rounding each; sim = 0 when either norm
    is 0;
  * the residual x - r (fp32, one rounding per element) is quantised by the
    int8 rule of cache.py; a reference is stored with q = 0, s = 0;
  * reconstruction x^ = bf16(r + float(q) s) (fp32 multiply, fp32 add, bf16
    round to nearest even); a token with no reference has r = 0, so its
    reconstruction is the plain int8 one;
  * release (before the write, as the paper orders it): every token about to
    be written drops its reference; a slot that no token refers to is free;
  * allocation: the pool has R_cap slots; new references, in ascending token
    order, take the free slots in ascending slot order; a reference that finds
    no free slot is not created, and it and every row of its run are stored as
    plain int8 (no reference).

Pins: tau above every similarity makes every written row a reference that
reconstructs exactly; seg_len 1 does the same; an empty pool is the plain int8
cache bit for bit; the residual error bound; reference counts equal the
number of tokens that refer to each slot; a hand-worked scan.
"""
from __future__ import annotations

import numpy as np

from . import cache
from .select import canonical_sum

F32 = np.float32


class Int8Cache:
    """The plain int8 per-token cache (cache.py) behind the common interface."""

    kind = "int8"

    def __init__(self, NT: int, D: int):
        self.q = np.zeros((NT, D), dtype=np.int8)
        self.s = np.zeros(NT, dtype=F32)

    def reconstruct_f32(self) -> np.ndarray:
        return (self.q.astype(F32) * self.s[:, None]).astype(F32)

    def reconstruct_bf16(self) -> np.ndarray:
        return cache.dequantize_rows(self.q, self.s)

    def write(self, rows, vals) -> bool:
        return cache.quant_scatter(np.asarray(vals, dtype=F32), rows, self.q, self.s)

    def copy(self):
        c = Int8Cache(*self.q.shape)
        c.q, c.s = self.q.copy(), self.s.copy()
        return c


class FullCache:
    """Rows kept in the compute precision (bf16 values in fp32 storage)."""

    kind = "bf16"

    def __init__(self, NT: int, D: int):
        self.v = np.zeros((NT, D), dtype=F32)

    def reconstruct_f32(self) -> np.ndarray:
        return self.v.copy()

    def reconstruct_bf16(self) -> np.ndarray:
        return self.v.copy()

    def write(self, rows, vals) -> bool:
        vals = np.asarray(vals, dtype=F32)
        self.v[np.asarray(rows)] = vals
        return bool((~np.isfinite(vals)).any())

    def copy(self):
        c = FullCache(*self.v.shape)
        c.v = self.v.copy()
        return c


def similarity(x: np.ndarray, r: np.ndarray) -> np.ndarray:
    """fp32 cosine similarity of the rows of x [R, D] with the rows of r [R, D]."""
    x = np.asarray(x, dtype=F32)
    r = np.asarray(r, dtype=F32)
    dot = canonical_sum((x * r).astype(F32))
    nx = canonical_sum((x * x).astype(F32))
    nr = canonical_sum((r * r).astype(F32))
    den = (np.sqrt(nx).astype(F32) * np.sqrt(nr).astype(F32)).astype(F32)
    out = np.zeros(len(dot), dtype=F32)
    ok = (nx > 0) & (nr > 0)
    with np.errstate(divide="ignore", invalid="ignore"):
        out[ok] = (dot[ok] / den[ok]).astype(F32)
    return out


class RefCache:
    """The reference-plus-int8-residual cache manager of Sec. 3.4."""

    kind = "ref"

    def __init__(self, NT: int, D: int, R_cap: int, seg_len: int, tau: float):
        self.NT, self.D, self.R_cap, self.seg_len, self.tau = NT, D, R_cap, seg_len, F32(tau)
        self.ref = np.full(NT, -1, dtype=np.int32)
        self.q = np.zeros((NT, D), dtype=np.int8)
        self.s = np.zeros(NT, dtype=F32)
        self.pool = np.zeros((R_cap, D), dtype=F32)
        self.refcount = np.zeros(R_cap, dtype=np.int32)

    def copy(self):
        c = RefCache(self.NT, self.D, self.R_cap, self.seg_len, float(self.tau))
        for k in ("ref", "q", "s", "pool", "refcount"):
            setattr(c, k, getattr(self, k).copy())
        return c

    def _r(self) -> np.ndarray:
        r = np.zeros((self.NT, self.D), dtype=F32)
        has = self.ref >= 0
        r[has] = self.pool[self.ref[has]]
        return r

    def reconstruct_f32(self) -> np.ndarray:
        qs = (self.q.astype(F32) * self.s[:, None]).astype(F32)
        return (self._r() + qs).astype(F32)

    def reconstruct_bf16(self) -> np.ndarray:
        return cache.round_bf16(self.reconstruct_f32())

    def scan(self, rows: np.ndarray, vals: np.ndarray) -> np.ndarray:
        """Position (in rows) of the reference of every written row; a row that
        is its own reference starts a new run."""
        n = len(rows)
        src = np.zeros(n, dtype=np.int64)
        jr = -1
        for j in range(n):
            if jr >= 0 and rows[j] // self.seg_len != rows[jr] // self.seg_len:
                jr = -1                                  # a new scan segment
            if jr >= 0 and similarity(vals[j:j + 1], vals[jr:jr + 1])[0] > self.tau:
                src[j] = jr
            else:
                src[j] = j
                jr = j
        return src

    def write(self, rows, vals) -> bool:
        rows = np.asarray(rows, dtype=np.int64)
        vals = np.asarray(vals, dtype=F32)
        # release: every token about to be written drops its reference
        for i in rows:
            if self.ref[i] >= 0:
                self.refcount[self.ref[i]] -= 1
        src = self.scan(rows, vals)
        # allocation: new references in token order take the free slots in slot order
        free = np.flatnonzero(self.refcount == 0)
        refs = np.flatnonzero(src == np.arange(len(rows)))
        slot = {int(j): (int(free[m]) if m < len(free) else -1) for m, j in enumerate(refs)}
        bad = False
        for j, i in enumerate(rows):
            jr = int(src[j])
            sl = slot[jr]
            if sl < 0:                                   # no slot: plain int8
                q, s, b = cache.quantize_rows(vals[j:j + 1])
                self.ref[i] = -1
            elif jr == j:                                # a new reference
                self.pool[sl] = vals[j]
                q, s, b = np.zeros((1, self.D), np.int8), np.zeros(1, F32), np.zeros(1, bool)
                self.ref[i] = sl
                self.refcount[sl] += 1
            else:                                        # int8 residual against it
                delta = (vals[j:j + 1] - vals[jr:jr + 1]).astype(F32)
                q, s, b = cache.quantize_rows(delta)
                self.ref[i] = sl
                self.refcount[sl] += 1
            self.q[i], self.s[i] = q[0], s[0]
            bad |= bool(b[0])
        return bad

    def stats(self) -> tuple[int, int]:
        """(live references, high-water mark = 1 + the highest live slot)."""
        live = np.flatnonzero(self.refcount > 0)
        return len(live), (int(live[-1]) + 1 if len(live) else 0)
