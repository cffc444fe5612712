"""CUDA path vs oracle, element by element, on small and ragged problems.

Every call goes through the C-ABI (ctypes binding).  Sizes span several
buckets / tiles and a ragged tail; the edge cases are d = 1, d < 32,
d not a multiple of 4, 32, the bucket or the top-k tile, zeros of both
signs, ties, k = 1 and k = d, non-power-of-two M, and the smallest and
largest buckets.
"""
from __future__ import annotations

import numpy as np
import pytest

import oracle
from parity_helpers import (STEP_RTOL, assert_bits_equal, assert_messages_equal, oracle_config,
                            assert_params_equal)

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def P():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2010_13359_gb300 as P
    return P


def gpu_config(P, ocfg, stream):
    return P.make_config(d=ocfg.d, M=ocfg.M, compressor=ocfg.compressor, lr=ocfg.lr, bucket=ocfg.bucket,
                         k=ocfg.k, bits=ocfg.bits, seed=ocfg.seed,
                         flags=P.KEEP_LOOKAHEAD if ocfg.keep_lookahead else 0,
                         cuda_stream=stream.cuda_stream)


def grads(kind, M, d, rng):
    if kind == "gauss":
        return (rng.standard_normal((M, d)) * np.exp(rng.uniform(-4, 1, (M, d)))).astype(np.float32)
    if kind == "ties":  # many exact ties, zeros of both signs
        g = (rng.integers(-2, 3, size=(M, d)) * 0.5).astype(np.float32)
        g[g == 0] = np.where(rng.random((g == 0).sum()) < 0.5, -0.0, 0.0)
        return g
    if kind == "zeros":
        return np.zeros((M, d), np.float32)
    raise ValueError(kind)


def run_parity(P, ocfg, T, kind="gauss", batched=True, seed=0):
    """T free-running steps on both sides; every step compares messages,
    e, h and w bit for bit (w also within STEP_RTOL per element)."""
    dev = torch.device("cuda:0")
    stream = torch.cuda.current_stream(dev)
    rng = np.random.default_rng(seed)
    h = P.create(gpu_config(P, ocfg, stream))
    st = oracle.State(ocfg)
    d, M = ocfg.d, ocfg.M
    mb = h.message_bytes()
    assert mb == oracle.message_bytes(ocfg)
    w0 = (rng.standard_normal(d) * 0.02).astype(np.float32)
    w_gpu = torch.from_numpy(w0.copy()).to(dev)
    w_orc = w0.copy()
    ld = (d + 3) // 4 * 4
    for t in range(1, T + 1):
        g = grads(kind, M, d, rng)
        g_dev = torch.zeros((M, ld), dtype=torch.float32, device=dev)
        g_dev[:, :d] = torch.from_numpy(g).to(dev)
        msgs = torch.zeros((M, mb), dtype=torch.uint8, device=dev)
        if ocfg.keep_lookahead:  # lookahead of every worker before the gradient
            for i in range(M):
                wh = torch.empty(d, dtype=torch.float32, device=dev)
                h.worker_lookahead(i, w_gpu, wh)
                assert_bits_equal(wh.cpu().numpy(), oracle.lookahead(w_orc, st.h[i]),
                                  f"lookahead worker {i} step {t}")
        if batched:
            h.workers_compress_all(g_dev, ld, msgs)
        else:
            for i in range(M):
                h.worker_compress(i, g_dev[i], msgs[i])
        msgs_orc = st.compress_all(g)
        got = msgs.cpu().numpy()
        for i in range(M):
            assert_messages_equal(ocfg, got[i], msgs_orc[i], f"worker {i} step {t}")
            e_i = np.empty(d, np.float32)
            h.get_residual(i, e_i)
            assert_bits_equal(e_i, st.e[i], f"residual worker {i} step {t}")
            if ocfg.keep_lookahead:
                h_i = np.empty(d, np.float32)
                h.get_lookahead(i, h_i)
                assert_bits_equal(h_i, st.h[i], f"lookahead offset worker {i} step {t}")
        h.server_aggregate_update(msgs, w_gpu)
        st.server(msgs_orc, w_orc)
        h.synchronize()
        assert_params_equal(w_gpu.cpu().numpy(), w_orc, f"params step {t}")
        assert h.get_step() == st.t == t + 1
    h.destroy()


EDGE_CASES = [
    (oracle.SIGN, dict(bucket=32)),
    (oracle.SIGN, dict(bucket=128)),
    (oracle.SIGN, dict(bucket=512)),
    (oracle.SIGN, dict(bucket=2048)),
    (oracle.SIGN, dict(bucket=4096)),
    (oracle.SQUANT, dict(bucket=32, bits=8)),
    (oracle.SQUANT, dict(bucket=64, bits=2)),
    (oracle.SQUANT, dict(bucket=512, bits=4)),
    (oracle.SQUANT, dict(bucket=4096, bits=8)),
    (oracle.QSGD, dict(bucket=32, bits=4)),
    (oracle.QSGD, dict(bucket=512, bits=8)),
    (oracle.QSGD, dict(bucket=4096, bits=2)),
    (oracle.TOPK, dict(k=1)),
    (oracle.TOPK, dict(k=7)),
    (oracle.TOPK, dict(k=-1)),  # k = d
    (oracle.IDENTITY, dict()),
]


def _case_id(c):
    comp, kw = c
    name = {0: "sign", 1: "topk", 2: "squant", 3: "identity", 4: "qsgd"}[comp]
    return name + "".join(f"-{k}{v}" for k, v in kw.items())


@pytest.mark.parametrize("case", EDGE_CASES, ids=_case_id)
@pytest.mark.parametrize("d", [1, 31, 33, 4100, 65537])
def test_edge_sizes(P, case, d):
    comp, kw = case
    kw = dict(kw)
    if comp == oracle.TOPK:
        kw["k"] = d if kw["k"] == -1 else min(kw["k"], d)
    ocfg = oracle_config(d, 3, comp, lr=0.05, seed=1234567, keep=True, **kw)
    run_parity(P, ocfg, T=3, seed=d)


@pytest.mark.parametrize("kind", ["ties", "zeros"])
@pytest.mark.parametrize("case", [(oracle.SIGN, dict(bucket=256)), (oracle.SQUANT, dict(bucket=256, bits=4)),
                                  (oracle.QSGD, dict(bucket=1024, bits=8)),
                                  (oracle.TOPK, dict(k=300)), (oracle.TOPK, dict(k=5000))], ids=_case_id)
def test_degenerate_values(P, case, kind):
    comp, kw = case
    ocfg = oracle_config(12_289, 2, comp, lr=1.0, seed=5, keep=True, **kw)
    run_parity(P, ocfg, T=3, kind=kind, seed=7)


@pytest.mark.parametrize("case", [(oracle.SIGN, dict(bucket=1024)), (oracle.SQUANT, dict(bucket=512, bits=8)),
                                  (oracle.QSGD, dict(bucket=2048, bits=4)),
                                  (oracle.TOPK, dict(k=2000)), (oracle.IDENTITY, dict())], ids=_case_id)
def test_per_worker_calls_match_batched(P, case):
    """dqgan_worker_compress per worker gives the same as the batched call."""
    comp, kw = case
    ocfg = oracle_config(200_003, 4, comp, lr=1e-2, seed=99, keep=True, **kw)
    run_parity(P, ocfg, T=2, batched=False, seed=3)


@pytest.mark.parametrize("M,comp,bucket", [
    (1, oracle.SIGN, 512), (5, oracle.SIGN, 512), (8, oracle.SIGN, 1024), (32, oracle.SIGN, 2048),
    (33, oracle.SIGN, 4096), (70, oracle.SIGN, 1024), (3, oracle.SIGN, 256), (40, oracle.SIGN, 64),
    (20, oracle.SQUANT, 512), (33, oracle.IDENTITY, 512), (9, oracle.TOPK, 512), (6, oracle.QSGD, 512),
    (40, oracle.QSGD, 1024)])
def test_worker_counts(P, M, comp, bucket):
    """Non-power-of-two M, M above 32 (several 32-worker slabs in the sign
    server), every server path."""
    ocfg = oracle_config(50_000 + 3, M, comp, lr=1e-2, bucket=bucket, bits=8, k=777)
    run_parity(P, ocfg, T=3, seed=M)


@pytest.mark.parametrize("M", [1, 7, 16, 17, 32])
@pytest.mark.parametrize("comp,bits,bucket", [(oracle.SQUANT, 2, 512), (oracle.SQUANT, 2, 1024),
                                              (oracle.QSGD, 2, 2048), (oracle.SQUANT, 4, 512)])
def test_squant_server_worker_counts(P, M, comp, bits, bucket):
    """The TMA quantiser servers at every worker count they take: b = 2 in
    one or two sets of 16 workers (pair tables, several slices per bucket),
    b = 4 by per-worker lookups; ragged last bucket."""
    ocfg = oracle_config(3 * 4096 + 2 * 512 + 100, M, comp, lr=1e-2, bucket=bucket, bits=bits, seed=M + bits)
    run_parity(P, ocfg, T=3, seed=M)


def test_multi_tile_topk_many_steps(P):
    """Top-k over many 4096-element tiles with a ragged last tile, 6 steps."""
    ocfg = oracle_config(3 * 4096 * 7 + 123, 3, oracle.TOPK, lr=0.1, k=1500, keep=True)
    run_parity(P, ocfg, T=6, seed=11)


def test_checkpoint_round_trip(P):
    """T steps straight through == T/2 steps, save, load into a new handle, T/2 steps."""
    dev = torch.device("cuda:0")
    stream = torch.cuda.current_stream(dev)
    ocfg = oracle_config(30_001, 3, oracle.SQUANT, lr=0.02, bucket=512, bits=4, seed=77, keep=True)
    rng = np.random.default_rng(0)
    G = [torch.from_numpy(grads("gauss", 3, ocfg.d, rng)).to(dev) for _ in range(6)]
    ld = ocfg.d

    def fresh():
        return P.create(gpu_config(P, ocfg, stream))

    w_a = torch.zeros(ocfg.d, device=dev)
    w_b = torch.zeros(ocfg.d, device=dev)
    a = fresh()
    mb = a.message_bytes()
    msgs = torch.zeros((3, mb), dtype=torch.uint8, device=dev)
    pad = torch.zeros((3, (ld + 3) // 4 * 4), device=dev)
    for t in range(6):
        pad[:, :ld] = G[t]
        a.workers_compress_all(pad, pad.shape[1], msgs)
        a.server_aggregate_update(msgs, w_a)
    b = fresh()
    for t in range(3):
        pad[:, :ld] = G[t]
        b.workers_compress_all(pad, pad.shape[1], msgs)
        b.server_aggregate_update(msgs, w_b)
    blob = np.zeros(b.state_bytes(), np.uint8)
    b.save_state(blob, blob.size)
    b.destroy()
    c = fresh()
    c.load_state(blob, blob.size)
    assert c.get_step() == 4
    for t in range(3, 6):
        pad[:, :ld] = G[t]
        c.workers_compress_all(pad, pad.shape[1], msgs)
        c.server_aggregate_update(msgs, w_b)
    c.synchronize()
    a.synchronize()
    assert torch.equal(w_a, w_b)
    for i in range(3):
        ea, ec = np.empty(ocfg.d, np.float32), np.empty(ocfg.d, np.float32)
        a.get_residual(i, ea)
        c.get_residual(i, ec)
        assert_bits_equal(ec, ea, "residual after resume")
    # a mismatching state is refused
    other = P.create(gpu_config(P, oracle_config(30_002, 3, oracle.SQUANT, bucket=512, bits=4, keep=True),
                                stream))
    with pytest.raises(P.DqganError) as ei:
        blob2 = np.zeros(other.state_bytes(), np.uint8)
        other.load_state(blob, blob2.size)
    assert ei.value.status == P.dqgan.ERR_INVALID_ARG
    for x in (a, c, other):
        x.destroy()


def test_error_conventions(P):
    dev = torch.device("cuda:0")
    stream = torch.cuda.current_stream(dev)
    h = P.create(P.make_config(d=1000, M=2, compressor=P.SIGN, bucket=128, cuda_stream=stream.cuda_stream))
    g = torch.zeros(1004, device=dev)
    msg = torch.zeros(h.message_bytes() + 16, dtype=torch.uint8, device=dev)
    with pytest.raises(P.DqganError) as ei:
        h.worker_compress(2, g, msg)  # worker out of range
    assert ei.value.status == P.dqgan.ERR_INVALID_ARG and "worker" in h.last_error()
    with pytest.raises(P.DqganError) as ei:
        h.worker_compress(0, g.data_ptr() + 4, msg)  # misaligned gradient
    assert ei.value.status == P.dqgan.ERR_INVALID_ARG
    with pytest.raises(P.DqganError) as ei:
        h.worker_compress(0, g, 0)  # NULL message
    assert ei.value.status == P.dqgan.ERR_INVALID_ARG
    with pytest.raises(P.DqganError) as ei:
        h.worker_lookahead(0, g, g)  # no KEEP_LOOKAHEAD
    assert ei.value.status == P.dqgan.ERR_UNSUPPORTED
    with pytest.raises(P.DqganError) as ei:
        h.workers_compress_all(g, 1002, msg)  # stride not a multiple of 4
    assert ei.value.status == P.dqgan.ERR_INVALID_ARG
    with pytest.raises(P.DqganError):
        h.set_step(0)
    before = h.launch_count()
    h.worker_compress(1, g, msg)
    assert h.launch_count() == before + 1
    h.synchronize()
    h.destroy()
    with pytest.raises(P.DqganError) as ei:
        P.create(P.make_config(d=0, M=2, compressor=P.SIGN))
    assert ei.value.status == P.dqgan.ERR_INVALID_ARG


@pytest.mark.parametrize("case", [(oracle.SIGN, dict(bucket=4096)), (oracle.SQUANT, dict(bucket=512, bits=8)),
                                  (oracle.TOPK, dict(k=999))], ids=_case_id)
def test_pinned_host_gradients_read_in_place(P, case):
    """Gradients in pinned host memory are read in place by the kernels (over
    the host link) and give the same bits as the same gradients in HBM."""
    comp, kw = case
    dev = torch.device("cuda:0")
    stream = torch.cuda.current_stream(dev)
    ocfg = oracle_config(100_003, 3, comp, lr=0.01, seed=5, **kw)
    ld = (ocfg.d + 3) // 4 * 4
    rng = np.random.default_rng(1)
    g_host = torch.zeros((ocfg.M, ld), dtype=torch.float32).pin_memory()
    g_host[:, :ocfg.d] = torch.from_numpy(grads("gauss", ocfg.M, ocfg.d, rng))
    g_dev = g_host.to(dev)
    a = P.create(gpu_config(P, ocfg, stream))
    b = P.create(gpu_config(P, ocfg, stream))
    mb = a.message_bytes()
    ma = torch.zeros((ocfg.M, mb), dtype=torch.uint8, device=dev)
    mbuf = torch.zeros((ocfg.M, mb), dtype=torch.uint8, device=dev)
    for _ in range(2):
        a.workers_compress_all(g_dev, ld, ma)
        b.workers_compress_all(g_host, ld, mbuf)
        a.synchronize()
        b.synchronize()
        assert torch.equal(ma, mbuf)
        for i in range(ocfg.M):
            ea, eb = np.empty(ocfg.d, np.float32), np.empty(ocfg.d, np.float32)
            a.get_residual(i, ea)
            b.get_residual(i, eb)
            assert_bits_equal(eb, ea, f"residual worker {i}")
    a.destroy()
    b.destroy()
