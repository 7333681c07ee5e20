"""A cached DiT stack driven through the C ABI: the user-facing step.

`CachedStack` owns the per-layer int8 caches, the workspaces and the index
buffers on the device and runs one denoising step as the paper orders it
(Sec. 3.3): the audio energy once per generation, then per layer the
energy-guided selection and the block on the selected latents.  Step 0 (or
any step with full=True) refreshes every token and fills the caches.  No host
synchronisation happens inside a step: K follows from the ratio on the host.
"""
from __future__ import annotations

import torch

from . import echocache as ec


class CachedStack:
    def __init__(self, T: int, N: int, D: int, H: int, d: int, F: int, Lc: int,
                 blocks: list, device="cuda", lam: float = 0.1, xi: float = 1e-6,
                 mode: int = ec.MODE_ENERGY_DRIFT):
        self.T, self.N, self.D = T, N, D
        self.NT = T * N
        self.dims = ec.BlockDims(T, N, D, H, d, F, Lc)
        self.blocks = blocks
        self.lam, self.xi, self.mode = lam, xi, mode
        dev = torch.device(device)
        L = len(blocks)
        self.cache_q = [torch.zeros(self.NT, D, dtype=torch.int8, device=dev) for _ in range(L)]
        self.cache_s = [torch.zeros(self.NT, dtype=torch.float32, device=dev) for _ in range(L)]
        self.ws = torch.empty(ec.echo_workspace_size(self.dims, self.NT), dtype=torch.uint8,
                              device=dev)
        self.sel_ws = torch.empty(ec.echo_select_workspace_size(T, N), dtype=torch.uint8, device=dev)
        self.idx = torch.empty(self.NT, dtype=torch.int32, device=dev)
        self.all_idx = torch.arange(self.NT, dtype=torch.int32, device=dev)
        self.scores = torch.empty(self.NT, dtype=torch.float32, device=dev)
        self.y = [torch.empty(self.NT, D, dtype=torch.bfloat16, device=dev) for _ in range(2)]
        self.band = torch.empty(T, 8, dtype=torch.float32, device=dev)
        self.seg = torch.zeros(T, dtype=torch.float32, device=dev)
        self.last_K = []

    def set_audio(self, audio: torch.Tensor, n_fft: int = 512, hop: int = 160, n_bands: int = 8):
        if self.band.shape[1] != n_bands:
            self.band = torch.empty(self.T, n_bands, dtype=torch.float32, device=self.seg.device)
        ec.echo_audio_energy(audio, self.T, n_fft, hop, n_bands, self.band, self.seg)
        return self.band, self.seg

    def step(self, x: torch.Tensor, ratio_num: int, ratio_den: int, full: bool = False,
             keep_scores: bool = False) -> torch.Tensor:
        """One denoising step over every layer; returns the last layer's output."""
        cur = x
        self.last_K = []
        for l, blk in enumerate(self.blocks):
            if full:
                idx, K = self.all_idx, self.NT
            else:
                idx, K, _ = ec.echo_select(cur, self.cache_q[l], self.cache_s[l], self.seg, self.T,
                                           self.N, ratio_num, ratio_den, self.lam, self.xi,
                                           self.mode, idx=self.idx,
                                           scores=self.scores if keep_scores else None,
                                           workspace=self.sel_ws)
            out = self.y[l % 2]
            ec.echo_block_step(blk, self.dims, cur, idx, K, self.cache_q[l], self.cache_s[l],
                               y=out, workspace=self.ws)
            self.last_K.append(K)
            cur = out
        return cur
