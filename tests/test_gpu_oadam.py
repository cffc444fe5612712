"""The Optimistic Adam server update (dqgan_set_server_optimizer) against the
oracle, element by element, through the C-ABI.

For every compressor and server kernel family (the scaled sign's table
kernels with flat and per-layer buckets, the b-bit quantisers, QSGD, the
identity, top-k), T free-running steps: messages bit for bit, then the
parameters w and the state m, v, u_prev bit for bit -- the update is fused
into the server kernel and both sides round every operation once in the
same order.  Also: the reduction setting (b1 = 0, identity preconditioner,
alpha = 1), a checkpoint round trip with the optimizer state, and the
argument checks.
"""
from __future__ import annotations

import numpy as np
import pytest

import oracle
from parity_helpers import assert_bits_equal, assert_messages_equal, assert_params_equal

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

ADAM = dict(alpha=1e-3, beta1=0.5, beta2=0.999, eps=1e-8, adaptive=True, bias_correction=True)
OMD_LIKE = dict(alpha=1.0, beta1=0.0, beta2=0.0, eps=0.0, adaptive=False, bias_correction=False)


@pytest.fixture(scope="module")
def P():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2010_13359_gb300 as P
    return P


def run(P, ocfg, opt_kw, T, segments=None, seed=0, env=None, monkeypatch=None):
    if env and monkeypatch:
        for k, v in env.items():
            monkeypatch.setenv(k, v)
    dev = torch.device("cuda:0")
    stream = torch.cuda.current_stream(dev)
    rng = np.random.default_rng(seed)
    d, M = ocfg.d, ocfg.M
    h = P.create(P.make_config(d=d, M=M, compressor=ocfg.compressor, lr=ocfg.lr, bucket=ocfg.bucket,
                               k=ocfg.k, bits=ocfg.bits, seed=ocfg.seed, cuda_stream=stream.cuda_stream))
    if segments is not None:
        h.set_segments(segments)
    h.set_server_optimizer(P.dqgan.oadam(**opt_kw))
    st = oracle.State(ocfg)
    opt = oracle.OAdamState(d, oracle.OAdam(**opt_kw))
    mb = h.message_bytes()
    w0 = (rng.standard_normal(d) * 0.02).astype(np.float32)
    w_gpu = torch.from_numpy(w0.copy()).to(dev)
    w_orc = w0.copy()
    ld = (d + 3) // 4 * 4
    g_dev = torch.zeros((M, ld), dtype=torch.float32, device=dev)
    msgs = torch.zeros((M, mb), dtype=torch.uint8, device=dev)
    for t in range(1, T + 1):
        g = (rng.standard_normal((M, d)) * np.exp(rng.uniform(-3, 1, (M, d)))).astype(np.float32)
        g_dev[:, :d] = torch.from_numpy(g).to(dev)
        h.workers_compress_all(g_dev, ld, msgs)
        h.server_aggregate_update(msgs, w_gpu)
        want = st.compress_all(g)
        got = msgs.cpu().numpy()
        for i in range(M):
            assert_messages_equal(ocfg, got[i], want[i], f"worker {i} step {t}")
        q_hat = oracle.server_average(ocfg, want)
        opt.update(t, q_hat, w_orc)
        st.t += 1
        assert_params_equal(w_gpu.cpu().numpy(), w_orc, f"step {t}")
        for which, ref in enumerate((opt.m, opt.v, opt.u)):
            buf = np.empty(d, np.float32)
            h.get_server_state(which, buf)
            assert_bits_equal(buf, ref, f"step {t} optimizer state {'mvu'[which]}")
    h.destroy()


CASES = [
    ("sign512", dict(d=20_011, M=5, compressor=oracle.SIGN, bucket=512)),
    ("sign4096_col", dict(d=1 << 22, M=8, compressor=oracle.SIGN, bucket=4096)),
    ("sign1024_tma", dict(d=100_003, M=32, compressor=oracle.SIGN, bucket=1024)),
    ("sign_slabs", dict(d=50_000, M=40, compressor=oracle.SIGN, bucket=512)),
    ("sign_small_bucket", dict(d=9_999, M=3, compressor=oracle.SIGN, bucket=64)),
    ("squant_b2", dict(d=123_457, M=16, compressor=oracle.SQUANT, bucket=512, bits=2)),
    ("squant_b4", dict(d=123_457, M=12, compressor=oracle.SQUANT, bucket=512, bits=4)),
    ("squant_b8", dict(d=123_457, M=20, compressor=oracle.SQUANT, bucket=512, bits=8)),
    ("squant_b8_many", dict(d=30_001, M=33, compressor=oracle.SQUANT, bucket=256, bits=8)),
    ("qsgd_b8", dict(d=77_777, M=7, compressor=oracle.QSGD, bucket=512, bits=8)),
    ("identity", dict(d=10_007, M=6, compressor=oracle.IDENTITY)),
    ("topk", dict(d=300_007, M=8, compressor=oracle.TOPK, k=3_000)),
    ("topk_one_worker", dict(d=5_003, M=1, compressor=oracle.TOPK, k=50)),
]


@pytest.mark.parametrize("name,kw", CASES, ids=[c[0] for c in CASES])
def test_oadam_server_matches_oracle(P, name, kw):
    ocfg = oracle.Config(lr=1e-2, seed=5, **kw)
    run(P, ocfg, ADAM, T=4)


@pytest.mark.parametrize("name,kw", [CASES[0], CASES[5], CASES[11]], ids=["sign", "squant_b2", "topk"])
def test_oadam_reduction_setting_matches_oracle(P, name, kw):
    ocfg = oracle.Config(lr=1e-2, seed=5, **kw)
    run(P, ocfg, OMD_LIKE, T=4)


@pytest.mark.parametrize("comp,bits", [(oracle.SIGN, 1), (oracle.SQUANT, 8)])
def test_oadam_with_layer_segments(P, comp, bits):
    d = 200_000
    segs = (0, 4_096, 70_016, 123_456 // 32 * 32, d)
    ocfg = oracle.Config(d=d, M=8, compressor=comp, bucket=1024, bits=bits, lr=1e-2, seed=9, segments=segs)
    run(P, ocfg, ADAM, T=3, segments=segs)


@pytest.mark.parametrize("path", ["col", "tma"])
def test_oadam_both_sign_server_kernels(P, path, monkeypatch):
    ocfg = oracle.Config(d=1_000_003, M=16, compressor=oracle.SIGN, bucket=2048, lr=1e-2, seed=3)
    run(P, ocfg, ADAM, T=3, env={"DQGAN_SIGN_SERVER": path}, monkeypatch=monkeypatch)


def test_oadam_checkpoint_round_trip(P):
    dev = torch.device("cuda:0")
    stream = torch.cuda.current_stream(dev)
    d, M = 40_000, 4
    cfg = P.make_config(d=d, M=M, compressor=P.SQUANT, bucket=512, bits=4, lr=1e-2, seed=2,
                        cuda_stream=stream.cuda_stream)
    rng = np.random.default_rng(1)
    gs = [torch.from_numpy((rng.standard_normal((M, d))).astype(np.float32)).to(dev) for _ in range(5)]
    w_a = torch.from_numpy((rng.standard_normal(d) * 0.02).astype(np.float32)).to(dev)
    w_b = w_a.clone()
    opt = P.dqgan.oadam(**ADAM)
    a = P.create(cfg)
    a.set_server_optimizer(opt)
    mb = a.message_bytes()
    msgs = torch.zeros((M, mb), dtype=torch.uint8, device=dev)
    for t in range(3):
        a.workers_compress_all(gs[t], d, msgs)
        a.server_aggregate_update(msgs, w_a)
    n = a.state_bytes()
    assert n == 64 + M * d * 4 + 3 * d * 4
    buf = np.zeros(n, np.uint8)
    a.save_state(buf, n)
    w_b.copy_(w_a)
    for t in range(3, 5):
        a.workers_compress_all(gs[t], d, msgs)
        a.server_aggregate_update(msgs, w_a)
    b = P.create(cfg)
    with pytest.raises(P.DqganError):  # the header says Optimistic Adam, the handle has the plain rule
        b.load_state(buf, n)
    b.set_server_optimizer(opt)
    b.load_state(buf, n)
    assert b.get_step() == 4
    for t in range(3, 5):
        b.workers_compress_all(gs[t], d, msgs)
        b.server_aggregate_update(msgs, w_b)
    assert torch.equal(w_a, w_b)
    for which in range(3):
        x, y = np.empty(d, np.float32), np.empty(d, np.float32)
        a.get_server_state(which, x)
        b.get_server_state(which, y)
        assert np.array_equal(x.view(np.uint32), y.view(np.uint32))
    a.destroy()
    b.destroy()


def test_oadam_argument_checks(P):
    dev = torch.device("cuda:0")
    stream = torch.cuda.current_stream(dev)
    mk = lambda **kw: P.create(P.make_config(cuda_stream=stream.cuda_stream, **kw))
    h = mk(d=1000, M=4, compressor=P.SIGN, bucket=512)
    buf = np.empty(1000, np.float32)
    with pytest.raises(P.DqganError) as ei:
        h.get_server_state(0, buf)
    assert ei.value.status == P.dqgan.ERR_UNSUPPORTED
    for bad in (dict(beta1=1.0), dict(beta2=-0.1), dict(eps=-1.0), dict(alpha=float("inf"))):
        kw = dict(ADAM)
        kw.update(bad)
        with pytest.raises(P.DqganError) as ei:
            h.set_server_optimizer(P.dqgan.oadam(**kw))
        assert ei.value.status == P.dqgan.ERR_INVALID_ARG
    h.set_server_optimizer(P.dqgan.oadam(**ADAM))
    with pytest.raises(P.DqganError) as ei:
        h.get_server_state(3, buf)
    assert ei.value.status == P.dqgan.ERR_INVALID_ARG
    g = torch.zeros((4, 1000), device=dev)
    msgs = torch.zeros((4, h.message_bytes()), dtype=torch.uint8, device=dev)
    w = torch.zeros(1000, device=dev)
    h.workers_compress_all(g, 1000, msgs)
    h.server_aggregate_update(msgs, w)
    with pytest.raises(P.DqganError) as ei:  # after the first step
        h.set_server_optimizer(P.dqgan.oadam(**ADAM))
    assert ei.value.status == P.dqgan.ERR_INVALID_ARG
    h.destroy()
    h = mk(d=1000, M=65, compressor=P.TOPK, k=10)
    with pytest.raises(P.DqganError) as ei:
        h.set_server_optimizer(P.dqgan.oadam(**ADAM))
    assert ei.value.status == P.dqgan.ERR_UNSUPPORTED
    h.destroy()
