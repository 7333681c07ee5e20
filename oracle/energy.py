"""Audio time-frequency energy -> per-segment saliency (Sec. 3.3, "Cross-modal Saliency Anchors").

TEST INFRASTRUCTURE ONLY (see the package header).

The paper splits the audio evenly into T segments, takes an STFT of each and
uses the L2 norm of each segment's time-frequency matrix as energy[tau].  It
gives neither window, hop, FFT size, padding nor bands; the readings used here:
  * segment length L_s = floor(L / T); the tail remainder is dropped;
  * inside a segment, frames start at 0, hop, 2 hop, ... while
    start + n_fft <= L_s; a segment shorter than n_fft gets one zero-padded frame;
  * periodic Hann window w[n] = 0.5 - 0.5 cos(2 pi n / n_fft), no centring;
  * one-sided power with Parseval weights: P_k = c_k |X_k|^2 / n_fft,
    c_0 = c_{n/2} = 1, other c_k = 2, so that sum_k P_k = sum_n (w[n] x[n])^2;
  * n_bands linear bands over the n_fft/2 + 1 bins, band b = [floor(B b / n_bands),
    floor(B (b + 1) / n_bands)) with B = n_fft/2 + 1;
  * band[tau, b] = sum over frames and bins of band b of P_k;
    energy[tau] = sqrt(sum_b band[tau, b])  (the norm of the segment's TF matrix).

The DFT is the plain definition X_k = sum_n w[n] x[n] exp(-2 pi i k n / n_fft),
evaluated in fp64 as a matrix product (one library matmul).

Pins: Parseval (band sum equals the windowed time-domain energy), one frame
against a library real FFT, silence gives exactly 0, a 440 Hz tone puts its
energy in band 0, homogeneity energy(c x) = |c| energy(x), frame counts.
"""
from __future__ import annotations

import numpy as np


def hann_periodic(n_fft: int) -> np.ndarray:
    n = np.arange(n_fft, dtype=np.float64)
    return 0.5 - 0.5 * np.cos(2.0 * np.pi * n / n_fft)


def segment_length(n_samples: int, T: int) -> int:
    return n_samples // T


def frame_offsets(seg_len: int, n_fft: int, hop: int) -> list[int]:
    if seg_len < n_fft:
        return [0]
    return list(range(0, seg_len - n_fft + 1, hop))


def band_edges(n_fft: int, n_bands: int) -> list[int]:
    n_bins = n_fft // 2 + 1
    return [(n_bins * b) // n_bands for b in range(n_bands + 1)]


def dft_power(frames: np.ndarray, n_fft: int) -> np.ndarray:
    """One-sided Parseval-weighted power P_k of windowed frames [n_frames, n_fft] (fp64)."""
    n = np.arange(n_fft, dtype=np.float64)
    k = np.arange(n_fft // 2 + 1, dtype=np.float64)
    ang = -2.0 * np.pi * np.outer(n, k) / n_fft
    X = frames @ (np.cos(ang) + 1j * np.sin(ang))
    c = np.full(n_fft // 2 + 1, 2.0)
    c[0] = 1.0
    c[-1] = 1.0
    return c * (X.real ** 2 + X.imag ** 2) / n_fft


def segment_frames(audio: np.ndarray, T: int, n_fft: int, hop: int) -> np.ndarray:
    """Windowed frames [T, n_frames, n_fft] following the segment-first order of Sec. 3.3."""
    a = np.asarray(audio, dtype=np.float64)
    Ls = segment_length(len(a), T)
    offs = frame_offsets(Ls, n_fft, hop)
    w = hann_periodic(n_fft)
    out = np.zeros((T, len(offs), n_fft))
    for tau in range(T):
        seg = a[tau * Ls:(tau + 1) * Ls]
        for f, o in enumerate(offs):
            piece = seg[o:o + n_fft]
            out[tau, f, :len(piece)] = piece * w[:len(piece)]
    return out


def audio_energy(audio: np.ndarray, T: int, n_fft: int = 512, hop: int = 160,
                 n_bands: int = 8):
    """Returns (band[T, n_bands], energy[T]) in fp64."""
    fr = segment_frames(audio, T, n_fft, hop)
    P = dft_power(fr.reshape(-1, n_fft), n_fft).reshape(T, fr.shape[1], -1)
    per_bin = P.sum(axis=1)                       # [T, n_bins], summed over frames
    e = band_edges(n_fft, n_bands)
    band = np.stack([per_bin[:, e[b]:e[b + 1]].sum(axis=1) for b in range(n_bands)], axis=1)
    energy = np.sqrt(band.sum(axis=1))
    return band, energy


def segment_weights(energy_f32: np.ndarray, lam: float) -> np.ndarray:
    """Per-segment saliency weight w_tau = lam + (1 - lam) * energy_tau / max energy.

    The paper turns energy into a top-k index set of high-energy segments
    (Sec. 3.3) but never gives k.  Reading: energy acts as a multiplicative
    weight on each token's drift, normalised by the largest segment energy, with
    a floor lam so that quiet segments can still be refreshed by drift.  All
    zero energy (silence) gives w = 1.  fp32 arithmetic in this order:
    t = e / e_max, w = lam + (1 - lam) * t.
    """
    e = np.asarray(energy_f32, dtype=np.float32)
    emax = np.float32(e.max()) if e.size else np.float32(0)
    if not emax > 0:
        return np.ones_like(e, dtype=np.float32)
    lam32 = np.float32(lam)
    one_minus = np.float32(np.float32(1.0) - lam32)
    t = (e / emax).astype(np.float32)
    return (lam32 + (one_minus * t).astype(np.float32)).astype(np.float32)
