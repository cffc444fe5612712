"""Algorithm 2 with the M simulated workers sharded over several GPUs.

With G ranks (one GPU each, one process per GPU), rank r owns the contiguous
workers [min(M, rR), min(M, (r+1)R)), R = ceil(M / G), and keeps only their
residuals (dqgan_set_local_workers).  One step of Algorithm 2 is then:

1. worker part: the rank's workers compress their gradients into the rank's
   R rows of a gather buffer (dqgan_workers_compress_range);
2. exchange: one all-gather of the packed messages over the process group
   (NCCL between GPUs) -- the workers' push to the server and the pull of
   the average (Section 2.3, Algorithm 2).  With this partition the first M
   rows of the gathered buffer are the M messages in worker order, the
   padding rows of the last ranks after them;
3. server part: every rank runs the same server step on its own replica of
   w (dqgan_server_aggregate_update).  The server's sum over workers has one
   fixed order, so the replicas stay equal bit for bit and no second
   collective is needed.

The compute goes through an engine with two calls, compress_range(first,
count, g, msgs) and server(msgs, w): `CudaEngine` is the C-ABI library; the
collective is torch.distributed's all_gather on whatever backend the
process group has.
"""
from __future__ import annotations

from . import dqgan


def worker_range(M: int, world: int, rank: int) -> tuple[int, int]:
    """[first, end) of the workers rank `rank` of `world` owns."""
    R = -(-M // world)
    return min(M, rank * R), min(M, (rank + 1) * R)


class CudaEngine:
    """The C-ABI handle of one rank, holding only its workers' state."""

    def __init__(self, cfg: dqgan.Config, first: int, count: int):
        self.h = dqgan.create(cfg)
        if count > 0:
            self.h.set_local_workers(first, count)

    def message_bytes(self) -> int:
        return self.h.message_bytes()

    def compress_range(self, first: int, count: int, g, g_stride: int, msgs) -> None:
        self.h.workers_compress_range(first, count, g, g_stride, msgs)

    def server(self, msgs, w) -> None:
        self.h.server_aggregate_update(msgs, w)

    def close(self) -> None:
        self.h.destroy()


class ShardedStep:
    """One rank's side of a sharded Algorithm 2 step (see the module text).

    engine: compress_range / server / message_bytes as `CudaEngine`;
    M: all workers; device: where the gather buffer lives (the engine's
    device for CUDA, "cpu" for a CPU process group); group: the process
    group (None: the default group, or a single process when
    torch.distributed is not initialised)."""

    def __init__(self, engine, M: int, device="cpu", group=None):
        import torch
        import torch.distributed as dist

        self.engine, self.M, self.group = engine, M, group
        self.dist = dist if dist.is_available() and dist.is_initialized() else None
        self.world = self.dist.get_world_size(group) if self.dist else 1
        self.rank = self.dist.get_rank(group) if self.dist else 0
        self.first, end = worker_range(M, self.world, self.rank)
        self.count = end - self.first
        self.R = -(-M // self.world)
        mb = engine.message_bytes()
        self.gather = torch.zeros((self.world * self.R, mb), dtype=torch.uint8, device=device)
        self.mine = self.gather[self.rank * self.R:(self.rank + 1) * self.R]
        self.parts = [self.gather[r * self.R:(r + 1) * self.R] for r in range(self.world)]
        self.msgs = self.gather[:M]

    def step(self, g_local, g_stride: int, w) -> None:
        """g_local: this rank's workers' gradients (row r: worker first + r)."""
        if self.count > 0:
            self.engine.compress_range(self.first, self.count, g_local, g_stride, self.mine)
        if self.dist and self.world > 1:
            self.dist.all_gather(self.parts, self.mine.clone(), group=self.group)
        self.engine.server(self.msgs, w)
