"""The sharded step of Algorithm 2 (paper_2010_13359_gb300/sharded.py) on CPU
ranks over gloo: world sizes 2 and 3, the M workers split unevenly, each
rank compressing only its own workers (here through the oracle, since this
container has no GPU: the engine is test scaffolding, the partition, the
gather buffer layout and the all-gather are the product's), then the
replicated server step.  Every rank's w must equal, bit for bit, a
single-process run of all M workers -- which also shows that the messages
really crossed between the ranks (a rank that saw only its own would
average zeros for the others)."""
from __future__ import annotations

import os
import socket

import numpy as np
import pytest

import oracle

torch = pytest.importorskip("torch")


class OracleEngine:
    """compress_range / server on the oracle, with the state of all M workers."""

    def __init__(self, cfg: oracle.Config):
        self.cfg = cfg
        self.st = oracle.State(cfg)

    def message_bytes(self):
        return oracle.message_bytes(self.cfg)

    def compress_range(self, first, count, g, g_stride, msgs):
        g = g.numpy() if hasattr(g, "numpy") else g
        for r in range(count):
            m = first + r
            msg = oracle.worker_step(self.cfg, m, self.st.t, g[r, :self.cfg.d], self.st.e[m])
            msgs[r].copy_(torch.from_numpy(msg))

    def server(self, msgs, w):
        oracle.server_step(self.cfg, msgs.numpy(), w.numpy())
        self.st.t += 1


def gradients(cfg, step, workers):
    rng = np.random.default_rng(1000 * step + 7)
    g = (rng.standard_normal((cfg.M, cfg.d)) * np.exp(rng.uniform(-3, 1, (cfg.M, cfg.d)))).astype(np.float32)
    return g[list(workers)]


def w0_of(cfg):
    return (np.random.default_rng(3).standard_normal(cfg.d) * 0.02).astype(np.float32)


def rank_main(rank, world, port, cfg, steps, out):
    import torch.distributed as dist

    from paper_2010_13359_gb300.sharded import ShardedStep, worker_range

    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        step = ShardedStep(OracleEngine(cfg), cfg.M, device="cpu")
        first, end = worker_range(cfg.M, world, rank)
        assert (step.first, step.first + step.count) == (first, end)
        w = torch.from_numpy(w0_of(cfg).copy())
        for t in range(1, steps + 1):
            g = torch.from_numpy(np.ascontiguousarray(gradients(cfg, t, range(first, end))))
            step.step(g, cfg.d, w)
        out[rank] = w.numpy().tobytes()
    finally:
        dist.destroy_process_group()


def free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


@pytest.mark.parametrize("world,cfg", [
    (2, oracle.Config(d=3001, M=5, compressor=oracle.SIGN, bucket=256, lr=0.01)),
    (3, oracle.Config(d=2048, M=7, compressor=oracle.SQUANT, bucket=512, bits=4, lr=0.01, seed=9)),
    (2, oracle.Config(d=4000, M=4, compressor=oracle.TOPK, k=40, lr=0.01)),
    (3, oracle.Config(d=999, M=2, compressor=oracle.IDENTITY, lr=0.01)),
])
def test_sharded_step_equals_one_process(world, cfg):
    import torch.multiprocessing as tmp

    steps = 3
    mgr = tmp.get_context("spawn").Manager()
    out = mgr.dict()
    tmp.spawn(rank_main, args=(world, free_port(), cfg, steps, out), nprocs=world, join=True)
    st = oracle.State(cfg)
    w = w0_of(cfg)
    for t in range(1, steps + 1):
        st.step(gradients(cfg, t, range(cfg.M)), w)
    for r in range(world):
        got = np.frombuffer(out[r], np.float32)
        assert np.array_equal(got.view(np.uint32), w.view(np.uint32)), f"rank {r}"


def test_worker_partition_covers_every_worker_once():
    from paper_2010_13359_gb300.sharded import worker_range
    for M in range(1, 40):
        for world in range(1, 9):
            ranges = [worker_range(M, world, r) for r in range(world)]
            covered = [m for a, b in ranges for m in range(a, b)]
            assert covered == list(range(M))
            R = -(-M // world)
            # every rank's rows start at rank * R: the first M gathered rows are the messages in order
            assert all(a == min(M, r * R) for r, (a, b) in enumerate(ranges))
