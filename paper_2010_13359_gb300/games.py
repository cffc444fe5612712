"""A min-max game driven through the full Algorithm 2 loop on the device.

Algorithm 2 needs the stochastic operator F(w_{t-1/2}^(m); xi) at every
worker's lookahead point.  For the GANs of Section 4 F is the generator and
discriminator gradient (the caller's model, outside this library); here it is
the bilinear game of Section 2.2, min_x max_y x^T D y, with the operator

    F(x, y) = (D y, -D x) + sigma * xi,

D a fixed positive diagonal.  Simultaneous gradient steps spiral away from the
equilibrium (0, 0) of this game; the optimistic step of Algorithm 2, which
evaluates F at the lookahead point, contracts toward it, also with compressed,
error-compensated messages.  F is a few tensor operations (it stands for the
user's model); every step of Algorithm 2 -- lookahead, error feedback,
compression, decode, average, update -- runs in the library's kernels.
"""
from __future__ import annotations

import dataclasses

from .workloads import game_diag_np, game_noise_np


@dataclasses.dataclass
class BilinearGame:
    d: int                 # even: w = [x, y], x and y of length d/2
    noise_std: float = 0.0
    seed: int = 7

    def __post_init__(self):
        if self.d <= 0 or self.d % 2:
            raise ValueError("the bilinear game needs an even, positive d")

    def operator(self, w, out, step: int, worker: int, D=None):
        """out = F(w) + sigma * xi_(step, worker) on w's device, in fp32 with one
        rounding per multiply and per add."""
        import torch
        half = self.d // 2
        if D is None:
            D = torch.from_numpy(game_diag_np(self.d, self.seed)).to(w.device)
        torch.mul(D, w[half:], out=out[:half])
        torch.mul(D, w[:half], out=out[half:])
        out[half:].neg_()
        if self.noise_std != 0.0:
            noise = game_noise_np(self.d, self.seed, step, worker, self.noise_std)
            out.add_(torch.from_numpy(noise).to(w.device, non_blocking=True))
        return out


def closed_loop(handle, game: BilinearGame, w, steps: int, lookahead: bool = True, step0: int = 1,
                on_step=None):
    """Runs `steps` iterations of Algorithm 2 on the device parameters `w`
    through the C-ABI: per worker the lookahead point w_half (or w itself when
    `lookahead` is False) and g = F(w_half; xi); then the batched worker step
    over all M workers and the fused server step.  The handle must keep the
    lookahead offsets when `lookahead` is True.  `on_step(t, w_half, g, msgs)`
    sees each step's intermediates before the server step."""
    import torch
    if lookahead and not (handle.cfg.flags & 1):
        raise ValueError("closed_loop with lookahead needs a handle created with KEEP_LOOKAHEAD")
    dev = w.device
    M, d = handle.cfg.M, game.d
    if handle.cfg.d != d:
        raise ValueError("handle and game disagree on d")
    ld = (d + 3) // 4 * 4
    g = torch.zeros((M, ld), dtype=torch.float32, device=dev)
    w_half = torch.empty((M, d), dtype=torch.float32, device=dev)
    msgs = torch.zeros((M, handle.message_bytes()), dtype=torch.uint8, device=dev)
    D = torch.from_numpy(game_diag_np(d, game.seed)).to(dev)
    for t in range(step0, step0 + steps):
        for i in range(M):
            if lookahead:
                handle.worker_lookahead(i, w, w_half[i])
            else:
                w_half[i].copy_(w)
            game.operator(w_half[i], g[i, :d], t, i, D=D)
        handle.workers_compress_all(g, ld, msgs)
        if on_step is not None:
            on_step(t, w_half, g, msgs)
        handle.server_aggregate_update(msgs, w)
    return w
