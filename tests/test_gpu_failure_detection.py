"""Failure detection on the GPU without a fault: a kernel whose wait can never
be satisfied gives up after its poll limit, the host sees DQGAN_ERR_TIMEOUT
at the next synchronize, and the handle and the CUDA context stay usable --
the next step still matches the oracle bit for bit."""
from __future__ import annotations

import time

import numpy as np
import pytest

import oracle
from parity_helpers import STEP_RTOL, assert_bits_equal, assert_messages_equal, oracle_config, assert_params_equal

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def P():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2010_13359_gb300 as P
    return P


@pytest.mark.parametrize("polls", [1, 4096, 0])
def test_bounded_wait_times_out_and_the_handle_survives(P, polls):
    dev = torch.device("cuda:0")
    stream = torch.cuda.current_stream(dev)
    d, M = 10_000, 3
    ocfg = oracle_config(d, M, oracle.SIGN, bucket=1024, lr=0.01, seed=4)
    h = P.create(P.make_config(d=d, M=M, compressor=oracle.SIGN, bucket=1024, lr=0.01, seed=4,
                               cuda_stream=stream.cuda_stream))
    rng = np.random.default_rng(1)
    g = rng.standard_normal((M, d)).astype(np.float32)
    w0 = rng.standard_normal(d).astype(np.float32)
    st = oracle.State(ocfg)
    w_orc = w0.copy()
    w_gpu = torch.from_numpy(w0.copy()).to(dev)
    g_dev = torch.from_numpy(g).to(dev)
    msgs = torch.empty((M, h.message_bytes()), dtype=torch.uint8, device=dev)

    # a first step, then the self-test, then the same kind of step again
    h.workers_compress_all(g_dev, d, msgs)
    h.server_aggregate_update(msgs, w_gpu)
    st.step(g, w_orc)
    h.synchronize()
    t0 = time.perf_counter()
    h.selftest_wait_timeout(polls)
    with pytest.raises(P.DqganError) as exc:
        h.synchronize()
    waited = time.perf_counter() - t0
    assert exc.value.status == P.ERR_TIMEOUT
    assert "bounded device-side wait" in h.last_error()
    assert waited < 30.0
    h.synchronize()  # the word was cleared: no stale time-out
    assert torch.cuda.is_available() and torch.ones(4, device=dev).sum().item() == 4.0

    h.workers_compress_all(g_dev, d, msgs)
    want = st.compress_all(g)
    got = msgs.cpu().numpy()
    for i in range(M):
        assert_messages_equal(ocfg, got[i], want[i], f"worker {i} after the time-out")
    h.server_aggregate_update(msgs, w_gpu)
    st.server(want, w_orc)
    h.synchronize()
    assert_params_equal(w_gpu.cpu().numpy(), w_orc, "params")
    e0 = np.empty(d, np.float32)
    h.get_residual(0, e0)
    assert_bits_equal(e0, st.e[0], "residual after the time-out")
    assert h.get_step() == 3
    h.destroy()


def test_selftest_rejects_polls_above_the_limit(P):
    h = P.create(P.make_config(d=64, M=1, compressor=oracle.IDENTITY))
    with pytest.raises(P.DqganError) as exc:
        h.selftest_wait_timeout((1 << 21) + 1)
    assert exc.value.status == P.dqgan.ERR_INVALID_ARG
    h.destroy()
