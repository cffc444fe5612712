"""The sharding calls on one GPU: handles that each hold a range of the
workers (dqgan_set_local_workers) and compress it into their rows of one
message buffer (dqgan_workers_compress_range), then each run the server
step on their own replica of w -- the ranks of a sharded step emulated in
one process, with the message buffer standing in for the all-gather (no
kernel waits on another).  Every replica must equal, bit for bit, the
single-handle run over all workers, and so must the residuals; the single-
process ShardedStep (world size 1) must as well."""
from __future__ import annotations

import numpy as np
import pytest

import oracle

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def P():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2010_13359_gb300 as P
    return P


CASES = [
    dict(d=1 << 20, M=8, compressor=oracle.SIGN, bucket=4096),
    dict(d=300_007, M=5, compressor=oracle.SQUANT, bucket=512, bits=4),
    dict(d=200_000, M=6, compressor=oracle.TOPK, k=2_000),
    dict(d=65_537, M=3, compressor=oracle.IDENTITY),
]


@pytest.mark.parametrize("kw", CASES, ids=["sign", "squant_b4", "topk", "identity"])
@pytest.mark.parametrize("ranks", [2, 3])
def test_ranges_match_the_single_handle(P, kw, ranks):
    from paper_2010_13359_gb300.sharded import worker_range
    dev = torch.device("cuda:0")
    stream = torch.cuda.current_stream(dev)
    d, M = kw["d"], kw["M"]
    cfg = P.make_config(lr=1e-2, seed=4, cuda_stream=stream.cuda_stream, **kw)
    ref = P.create(cfg)
    mb = ref.message_bytes()
    parts = []
    for r in range(ranks):
        a, b = worker_range(M, ranks, r)
        h = P.create(cfg)
        if b > a:
            h.set_local_workers(a, b - a)
        parts.append((h, a, b))
    rng = np.random.default_rng(11)
    w0 = torch.from_numpy((rng.standard_normal(d) * 0.02).astype(np.float32)).to(dev)
    w_ref = w0.clone()
    w_rep = [w0.clone() for _ in range(ranks)]
    msgs_ref = torch.zeros((M, mb), dtype=torch.uint8, device=dev)
    msgs = torch.zeros((M, mb), dtype=torch.uint8, device=dev)
    ld = (d + 3) // 4 * 4  # gradient rows 16-byte aligned
    g = torch.zeros((M, ld), dtype=torch.float32, device=dev)
    for t in range(4):
        g[:, :d] = torch.from_numpy((rng.standard_normal((M, d)) * np.exp(rng.uniform(-3, 1, (M, d))))
                                    .astype(np.float32)).to(dev)
        ref.workers_compress_all(g, ld, msgs_ref)
        ref.server_aggregate_update(msgs_ref, w_ref)
        for h, a, b in parts:
            if b > a:
                h.workers_compress_range(a, b - a, g[a:b], ld, msgs[a:b])
        for (h, a, b), w in zip(parts, w_rep):
            h.server_aggregate_update(msgs, w)
        torch.cuda.synchronize(dev)
        assert torch.equal(msgs, msgs_ref), f"step {t}: messages"
        for r, w in enumerate(w_rep):
            assert torch.equal(w.view(torch.int32), w_ref.view(torch.int32)), f"step {t}: replica {r}"
    for h, a, b in parts:
        for i in range(a, b):
            x, y = np.empty(d, np.float32), np.empty(d, np.float32)
            h.get_residual(i, x)
            ref.get_residual(i, y)
            assert np.array_equal(x.view(np.uint32), y.view(np.uint32)), f"residual {i}"
        if b > a and a > 0:
            with pytest.raises(P.DqganError):  # outside the handle's range
                h.get_residual(a - 1, np.empty(d, np.float32))
            with pytest.raises(P.DqganError):  # not all workers are local
                h.workers_compress_all(g, ld, msgs)
        h.destroy()
    ref.destroy()


def test_sharded_step_single_process(P):
    from paper_2010_13359_gb300.sharded import CudaEngine, ShardedStep
    dev = torch.device("cuda:0")
    stream = torch.cuda.current_stream(dev)
    d, M = 123_456, 4
    cfg = P.make_config(d=d, M=M, compressor=P.SIGN, bucket=1024, lr=1e-2, cuda_stream=stream.cuda_stream)
    eng = CudaEngine(cfg, 0, M)
    step = ShardedStep(eng, M, device=dev)
    ref = P.create(cfg)
    msgs = torch.zeros((M, ref.message_bytes()), dtype=torch.uint8, device=dev)
    rng = np.random.default_rng(5)
    w0 = torch.from_numpy((rng.standard_normal(d) * 0.02).astype(np.float32)).to(dev)
    w_a, w_b = w0.clone(), w0.clone()
    for _ in range(3):
        g = torch.from_numpy(rng.standard_normal((M, d)).astype(np.float32)).to(dev)
        step.step(g, d, w_a)
        ref.workers_compress_all(g, d, msgs)
        ref.server_aggregate_update(msgs, w_b)
    torch.cuda.synchronize(dev)
    assert torch.equal(w_a.view(torch.int32), w_b.view(torch.int32))
    eng.close()
    ref.destroy()


def test_local_workers_checkpoint_round_trip(P):
    dev = torch.device("cuda:0")
    stream = torch.cuda.current_stream(dev)
    d, M = 50_000, 6
    cfg = P.make_config(d=d, M=M, compressor=P.SQUANT, bucket=512, bits=8, lr=1e-2, seed=1,
                        cuda_stream=stream.cuda_stream)
    a = P.create(cfg)
    a.set_local_workers(2, 3)
    n = a.state_bytes()
    assert n == 64 + 3 * d * 4
    rng = np.random.default_rng(2)
    msgs = torch.zeros((M, a.message_bytes()), dtype=torch.uint8, device=dev)
    g = torch.from_numpy(rng.standard_normal((3, d)).astype(np.float32)).to(dev)
    a.workers_compress_range(2, 3, g, d, msgs[2:5])
    buf = np.zeros(n, np.uint8)
    a.save_state(buf, n)
    b = P.create(cfg)
    with pytest.raises(P.DqganError):  # b holds all six workers: the state of three does not fit it
        b.load_state(buf, n)
    b.set_local_workers(2, 3)
    b.load_state(buf, n)
    for i in range(2, 5):
        x, y = np.empty(d, np.float32), np.empty(d, np.float32)
        a.get_residual(i, x)
        b.get_residual(i, y)
        assert np.array_equal(x.view(np.uint32), y.view(np.uint32))
    a.destroy()
    b.destroy()
