"""Pins for the oracle's int8 per-token cache (Sec. 3.4)."""
import numpy as np
import pytest

from oracle import cache as C
from synth import generate as G

F32 = np.float32


@pytest.mark.parametrize("seed,scale", [(0, 1.0), (1, 1e-3), (2, 300.0), (3, 1e-30)])
def test_quant_error_bound(seed, scale):
    v = G.random_rows(64, 256, seed=seed, scale=1.0) * F32(scale)
    q, s, bad = C.quantize_rows(v)
    assert not bad.any()
    err = np.abs(v.astype(np.float64) - q.astype(np.float64) * s[:, None].astype(np.float64))
    bound = s.astype(np.float64)[:, None] * (0.5 + 2.0 ** -14)
    assert (err <= bound).all()


def test_zero_row_gives_zero_scale_and_codes():
    v = np.zeros((3, 16), dtype=F32)
    v[1, 4] = 3.0
    q, s, bad = C.quantize_rows(v)
    assert s[0] == 0 and s[2] == 0 and not q[0].any() and not q[2].any()
    assert q[1, 4] == 127 and s[1] == F32(3.0) / F32(127.0)


def test_symmetry_and_extremes():
    v = G.random_rows(32, 64, seed=9)
    q, s, _ = C.quantize_rows(v)
    qn, sn, _ = C.quantize_rows(-v)
    assert np.array_equal(qn, -q) and np.array_equal(sn, s)
    amax_pos = np.abs(v).argmax(axis=1)
    assert (np.abs(q[np.arange(32), amax_pos]) == 127).all()
    assert q.min() >= -127 and q.max() <= 127


def test_hand_worked_rounding():
    # a = 127 gives s = 1 and inv = 1, so q = round_half_even(v)
    v = np.array([[127.0, -63.5, 0.5, 1.5, 2.5, -0.5, 3.25, 0.0]], dtype=F32)
    q, s, _ = C.quantize_rows(v)
    assert s[0] == 1.0
    assert list(q[0]) == [127, -64, 0, 2, 2, 0, 3, 0]


def test_nonfinite_row_is_flagged():
    v = np.ones((2, 8), dtype=F32)
    v[1, 2] = np.inf
    q, s, bad = C.quantize_rows(v)
    assert list(bad) == [False, True] and not q[1].any()


def test_bf16_round_nearest_even():
    # bf16 keeps 8 significant bits: around 1.0 the spacing is 2^-7.
    vals = np.array([1.0 + 2.0 ** -8,          # halfway, even neighbour is 1.0
                     1.0 + 3 * 2.0 ** -8,      # halfway, even neighbour is 1 + 2^-6
                     1.0 + 2.0 ** -8 + 2.0 ** -20,   # just above halfway -> up
                     -(1.0 + 2.0 ** -8),
                     3.40e38], dtype=F32)
    got = C.round_bf16(vals)
    assert got[0] == 1.0
    assert got[1] == F32(1.0 + 2.0 ** -6)
    assert got[2] == F32(1.0 + 2.0 ** -7)
    assert got[3] == -1.0
    assert np.isinf(got[4])


def test_dequant_is_bf16_of_fp32_product():
    q = np.array([[1, -1, 127, 0]], dtype=np.int8)
    s = np.array([1.0 + 3 * 2.0 ** -8], dtype=F32)
    got = C.dequantize_rows(q, s)
    assert got[0, 0] == F32(1.0 + 2.0 ** -6) and got[0, 1] == -got[0, 0] and got[0, 3] == 0
    # 127 * s = 127 + 381/256 = 128.48828125 exactly in fp32; bf16 spacing at 128 is 1
    assert got[0, 2] == 128.0


def test_quant_then_dequant_round_trip_error():
    v = G.random_rows(16, 512, seed=21)
    q, s, _ = C.quantize_rows(v)
    r = C.dequantize_rows(q, s).astype(np.float64)
    # quantisation error s/2 plus the bf16 rounding of the reconstruction
    bound = s[:, None] * (0.5 + 2.0 ** -14) + np.abs(r) * 2.0 ** -8
    assert (np.abs(r - v) <= bound).all()


def test_scatter_and_gather_rows():
    src = G.random_rows(3, 16, seed=4)
    qc = np.zeros((6, 16), dtype=np.int8)
    sc = np.zeros(6, dtype=F32)
    C.quant_scatter(src, [5, 0, 2], qc, sc)
    q, s, _ = C.quantize_rows(src)
    assert np.array_equal(qc[[5, 0, 2]], q) and not qc[[1, 3, 4]].any()
    assert np.array_equal(C.dequant_gather(qc, sc, [2, 5]), C.dequantize_rows(q[[2, 0]], s[[2, 0]]))
