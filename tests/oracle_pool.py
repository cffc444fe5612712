"""Per-worker oracle trajectories in worker processes (test infrastructure).

The workers of Algorithm 2 are independent until the server step, so each
worker's whole trajectory -- its messages at every step and its final
residual -- can be computed in its own process, from the same seeded numpy
gradients the GPU side is fed.  Pools must use the "spawn" start method.
"""
from __future__ import annotations

import numpy as np


def worker_trajectory(args):
    """(workload, overrides, worker, steps) -> (messages [steps x bytes], final e)."""
    import oracle
    from paper_2010_13359_gb300.workloads import WORKLOADS

    name, overrides, worker, steps = args
    wl = WORKLOADS[name].replace(**overrides)
    cfg = oracle.Config(d=wl.d, M=wl.M, compressor=wl.compressor, lr=wl.lr, bucket=wl.bucket, k=wl.k,
                        bits=wl.bits, seed=wl.seed)
    e = np.zeros(wl.d, np.float32)
    msgs = np.zeros((steps, oracle.message_bytes(cfg)), np.uint8)
    for t in range(1, steps + 1):
        g = wl.gradient_np(t, worker)
        msgs[t - 1] = oracle.worker_step(cfg, worker, t, g, e)
    return msgs, e
