"""Pins for the oracle's segment STFT energy (Sec. 3.3, "Cross-modal Saliency Anchors")."""
import numpy as np
import pytest

from oracle import energy as E
from synth import ALL, generate as G


def test_hann_is_periodic():
    w = E.hann_periodic(512)
    assert w[0] == 0.0 and w[256] == 1.0
    assert np.allclose(w[1:], w[1:][::-1], atol=1e-15, rtol=1e-12)


def test_band_edges_cover_all_bins():
    assert E.band_edges(512, 8) == [0, 32, 64, 96, 128, 160, 192, 224, 257]


@pytest.mark.parametrize("name,frames", [("tiny_256", 22), ("stack4_7800", 37),
                                         ("wan_block_32760", 21), ("wan_sweep_63960", 22)])
def test_frames_per_segment(name, frames):
    w = ALL[name]
    Ls = E.segment_length(w.n_samples, w.T)
    # closed form: floor((L_s - n_fft) / hop) + 1 frames fit in a segment
    assert len(E.frame_offsets(Ls, w.n_fft, w.hop)) == frames == (Ls - 512) // 160 + 1


def test_short_segment_gets_one_padded_frame():
    assert E.frame_offsets(300, 512, 160) == [0]
    a = np.ones(600, dtype=np.float32)
    band, e = E.audio_energy(a, 2)
    # Parseval on the zero-padded frame: sum of w[n]^2 over the 300 real samples
    w = E.hann_periodic(512)[:300]
    assert np.allclose(band.sum(axis=1), (w ** 2).sum(), rtol=1e-12)


def test_parseval_band_sum_equals_time_domain_energy():
    g = np.random.default_rng(7)
    a = g.standard_normal(16000).astype(np.float32)
    band, e = E.audio_energy(a, 4)
    Ls, w = 4000, E.hann_periodic(512)
    for tau in range(4):
        seg = a[tau * Ls:(tau + 1) * Ls].astype(np.float64)
        td = sum(float(((seg[o:o + 512] * w) ** 2).sum()) for o in range(0, Ls - 511, 160))
        assert abs(band[tau].sum() - td) <= 1e-12 * td
        assert abs(e[tau] - np.sqrt(td)) <= 1e-12 * np.sqrt(td)


def test_one_frame_matches_library_rfft():
    g = np.random.default_rng(3)
    a = g.standard_normal(512)
    band, _ = E.audio_energy(a, 1)
    X = np.fft.rfft(a * E.hann_periodic(512))
    c = np.full(257, 2.0)
    c[0] = c[-1] = 1.0
    P = c * np.abs(X) ** 2 / 512
    ref = [P[lo:hi].sum() for lo, hi in zip(E.band_edges(512, 8)[:-1], E.band_edges(512, 8)[1:])]
    assert np.allclose(band[0], ref, rtol=1e-11, atol=0)


def test_hann_cosine_at_bin_closed_form():
    # x[n] = cos(2 pi k0 n / N) under a periodic Hann window has X_k0 = N/4 and
    # X_{k0 +- 1} = -N/8, zero elsewhere; with P_k = 2|X_k|^2 / N that is N/8 at k0
    # and N/32 at the two neighbours.
    N, k0 = 512, 40
    n = np.arange(N)
    fr = (np.cos(2 * np.pi * k0 * n / N) * E.hann_periodic(N))[None, :]
    P = E.dft_power(fr, N)[0]
    expect = np.zeros(257)
    expect[k0] = N / 8
    expect[k0 - 1] = expect[k0 + 1] = N / 32
    assert np.allclose(P, expect, atol=1e-9)


def test_silence_is_exactly_zero_and_weights_are_one():
    w = ALL["tiny_256"]
    band, e = E.audio_energy(G.audio(w, "silence"), w.T)
    assert (band == 0).all() and (e == 0).all()
    assert (E.segment_weights(e.astype(np.float32), 0.1) == 1).all()


def test_tone_energy_sits_in_band_zero():
    w = ALL["tiny_256"]
    band, e = E.audio_energy(G.audio(w, "tone"), w.T)
    assert (band[:, 0] / band.sum(axis=1) > 1 - 1e-9).all()
    # closed form: a 0.5-amplitude sinusoid has mean square 1/8; a periodic Hann
    # window has mean square 3/8, so each frame carries about 512 * 3/64 energy
    per_frame = 512 * (3.0 / 8.0) * 0.125
    assert np.allclose(band.sum(axis=1) / 22, per_frame, rtol=2e-3)


def test_homogeneity_and_segment_locality():
    g = np.random.default_rng(11)
    a = g.standard_normal(8000)
    _, e = E.audio_energy(a, 4)
    _, e3 = E.audio_energy(-3.0 * a, 4)
    assert np.allclose(e3, 3 * e, rtol=1e-12)
    b = a.copy()
    b[2 * 2000:3 * 2000] *= 5.0
    _, eb = E.audio_energy(b, 4)
    assert np.array_equal(eb[[0, 1, 3]], e[[0, 1, 3]])
    assert eb[2] > 4.9 * e[2]


def test_segment_weights_rule():
    e = np.array([2.0, 8.0, 0.0, 4.0], dtype=np.float32)
    w = E.segment_weights(e, 0.1)
    assert w.dtype == np.float32
    assert w[1] == np.float32(1.0)           # the loudest segment gets weight 1
    assert w[2] == np.float32(0.1)           # silence keeps the floor lam
    # fp32 order: t = e/e_max, w = lam + (1-lam) t
    t = np.float32(2.0) / np.float32(8.0)
    assert w[0] == np.float32(0.1) + (np.float32(1.0) - np.float32(0.1)) * t
    assert w[0] < w[3] < w[1]
