"""Workload shapes for the energy-guided cached DiT step.

Shapes only: no arithmetic of the method lives here.  Token layout follows the
paper's notation (Sec. 3.1 "Preliminary" and Sec. 3.3 "Fine-grained latent-level
caching"): T temporal latent segments, N spatial latents per temporal position,
NT = T * N tokens of width D.  Heads H of size d (D = H * d), FFN width F, L_c
audio condition tokens, refresh ratio r = ratio_num / ratio_den.
"""
from __future__ import annotations

from dataclasses import dataclass, field, replace


@dataclass(frozen=True)
class Workload:
    name: str
    T: int            # latent frames = temporal segments
    Hp: int           # latent height after patching
    Wp: int           # latent width after patching
    D: int            # hidden size
    H: int            # attention heads
    d: int            # head dim
    F: int            # FFN width
    Lc: int           # audio condition tokens
    n_samples: int    # audio samples at 16 kHz
    ratio_num: int    # refresh ratio numerator
    ratio_den: int    # refresh ratio denominator
    steps: int = 1
    layers: int = 1
    sample_rate: int = 16000
    n_fft: int = 512
    hop: int = 160
    n_bands: int = 8
    profile: str = "speech"
    sweep_ratios: tuple = field(default_factory=tuple)
    sweep_profiles: tuple = field(default_factory=tuple)

    @property
    def N(self) -> int:
        return self.Hp * self.Wp

    @property
    def NT(self) -> int:
        return self.T * self.N

    @property
    def K(self) -> int:
        """Refresh budget ceil(r * NT), integer arithmetic only."""
        return (self.ratio_num * self.NT + self.ratio_den - 1) // self.ratio_den

    def with_ratio(self, num: int, den: int) -> "Workload":
        return replace(self, ratio_num=num, ratio_den=den)

    def with_profile(self, profile: str) -> "Workload":
        return replace(self, profile=profile)


# 4x8x8 latents, hidden 128, 2 heads x 64, FFN 512, 1 s of audio, 8 steps, r = 1/4.
TINY_256 = Workload("tiny_256", T=4, Hp=8, Wp=8, D=128, H=2, d=64, F=512, Lc=32,
                    n_samples=16000, ratio_num=1, ratio_den=4, steps=8, layers=1)

# 5x30x52 latents, hidden 1024, 16 heads x 64, FFN 4096, 2 s of audio,
# 4 blocks x 10 steps, r = 1/5.
STACK4_7800 = Workload("stack4_7800", T=5, Hp=30, Wp=52, D=1024, H=16, d=64, F=4096,
                       Lc=160, n_samples=32000, ratio_num=1, ratio_den=5, steps=10,
                       layers=4)

# Wan2.2-S2V-shaped block: 81 frames at 480x832 -> 21x30x52 latents, hidden 5120,
# 40 heads x 128, FFN 13824, 5.06 s of audio -> 672 condition tokens, r = 1/5.
WAN_BLOCK_32760 = Workload("wan_block_32760", T=21, Hp=30, Wp=52, D=5120, H=40, d=128,
                           F=13824, Lc=672, n_samples=80960, ratio_num=1, ratio_den=5,
                           steps=1, layers=1)

# The same block stacked 40 deep, 20 steps, refresh applied per step and per layer.
WAN_STACK40_32760 = replace(WAN_BLOCK_32760, name="wan_stack40_32760", steps=20, layers=40)

# 161 frames -> 41x30x52 = 63960 tokens; ratio and audio-profile sweep.
WAN_SWEEP_63960 = Workload("wan_sweep_63960", T=41, Hp=30, Wp=52, D=5120, H=40, d=128,
                           F=13824, Lc=672, n_samples=161000, ratio_num=1, ratio_den=5,
                           steps=1, layers=1,
                           sweep_ratios=((1, 20), (1, 10), (1, 5), (1, 2), (1, 1)),
                           sweep_profiles=("silence", "tone", "speech", "beats"))

ALL = {w.name: w for w in (TINY_256, STACK4_7800, WAN_BLOCK_32760, WAN_STACK40_32760,
                           WAN_SWEEP_63960)}


def small(name: str = "mini", T: int = 3, Hp: int = 4, Wp: int = 5, D: int = 64, H: int = 2,
          d: int = 32, F: int = 128, Lc: int = 8, n_samples: int = 4800, ratio_num: int = 1,
          ratio_den: int = 3, steps: int = 3, layers: int = 2) -> Workload:
    """A hand-sized workload for CPU-only checks."""
    return Workload(name, T=T, Hp=Hp, Wp=Wp, D=D, H=H, d=d, F=F, Lc=Lc,
                    n_samples=n_samples, ratio_num=ratio_num, ratio_den=ratio_den,
                    steps=steps, layers=layers)
