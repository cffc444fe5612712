"""dqgan_topk_compress_noalloc against the handle-based top-k path.

The no-allocation entry point serves callers that cannot allocate device
memory (and so cannot create a handle): it keeps its scratch in a fixed
array inside the library and works on a residual the caller owns.  It must
produce exactly the messages and residuals of dqgan_worker_compress with the
top-k compressor.  Four calls in a row, the last two with the gradient
scale dropped by 1e4 and then raised by 1e8, check that the shared scratch
is cleared between calls, that the caller's residual carries over, and that
the candidate threshold carried from call to call (also across the
parametrised cases, which share the array) never changes a result.
"""
from __future__ import annotations

import numpy as np
import pytest

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def P():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2010_13359_gb300 as P
    return P


@pytest.mark.parametrize("d,k", [(300_007, 3_000), (1 << 20, 10_486), (4_100, 4_100)])
def test_noalloc_topk_matches_handle_path(P, d, k):
    dev = torch.device("cuda:0")
    stream = torch.cuda.current_stream(dev)
    lr = 0.01
    h = P.create(P.make_config(d=d, M=1, compressor=P.TOPK, k=k, lr=lr, cuda_stream=stream.cuda_stream))
    mb = h.message_bytes()
    pad = (d + 3) // 4 * 4
    e_caller = torch.zeros(pad, dtype=torch.float32, device=dev)
    rng = np.random.default_rng(d)
    for call, scale in enumerate([1.0, 1.0, 1e-4, 1e4]):
        g = torch.zeros(pad, dtype=torch.float32, device=dev)
        g[:d] = torch.from_numpy((rng.standard_normal(d) * np.exp(rng.uniform(-3, 1, d)) * scale)
                                 .astype(np.float32))
        msg_ref = torch.zeros(mb, dtype=torch.uint8, device=dev)
        msg_new = torch.zeros(mb, dtype=torch.uint8, device=dev)
        h.worker_compress(0, g, msg_ref)
        P.dqgan.topk_compress_noalloc(g, e_caller, msg_new, d, k, lr, stream.cuda_stream)
        torch.cuda.synchronize(dev)
        assert torch.equal(msg_new[:8 * k], msg_ref[:8 * k]), f"call {call}: messages differ"
        e_ref = np.empty(d, np.float32)
        h.get_residual(0, e_ref)
        got = e_caller[:d].cpu().numpy()
        assert np.array_equal(got.view(np.uint32), e_ref.view(np.uint32)), f"call {call}: residuals differ"
        h.set_step(h.get_step() + 1)
    h.destroy()


def test_noalloc_exact_size_views_odd_d(P):
    """g and e are views of exactly d floats at an odd d, with guard words
    on both sides inside the same allocation: the scalar tail path must
    neither read past d (NaN guards would reach the selection and change the
    records against the oracle) nor write outside [0, d) of e."""
    import oracle
    dev = torch.device("cuda:0")
    stream = torch.cuda.current_stream(dev)
    d, k, lr, lead, tail = 300_007, 2_999, 0.01, 16, 61
    guard = np.float32(np.nan)
    g_buf = torch.full((lead + d + tail,), float(guard), dtype=torch.float32, device=dev)
    e_buf = torch.full((lead + d + tail,), float(guard), dtype=torch.float32, device=dev)
    g, e = g_buf[lead:lead + d], e_buf[lead:lead + d]
    assert g.data_ptr() % 16 == 0 and e.data_ptr() % 16 == 0
    e.zero_()
    e_orc = np.zeros(d, np.float32)
    cfg = oracle.Config(d=d, M=1, compressor=oracle.TOPK, lr=lr, k=k)
    rng = np.random.default_rng(7)
    msg = torch.zeros(8 * k, dtype=torch.uint8, device=dev)
    for call in range(2):
        g_host = (rng.standard_normal(d) * np.exp(rng.uniform(-3, 1, d))).astype(np.float32)
        g.copy_(torch.from_numpy(g_host))
        P.dqgan.topk_compress_noalloc(g, e, msg, d, k, lr, stream.cuda_stream)
        torch.cuda.synchronize(dev)
        want = oracle.worker_step(cfg, 0, call + 1, g_host, e_orc)
        assert np.array_equal(msg.cpu().numpy(), want[:8 * k]), f"call {call}: records differ from the oracle"
        assert np.array_equal(e.cpu().numpy().view(np.uint32), e_orc.view(np.uint32)), f"call {call}: residual"
        for name, buf in (("g", g_buf), ("e", e_buf)):
            host = buf.cpu().numpy()
            assert np.isnan(host[:lead]).all() and np.isnan(host[lead + d:]).all(), f"{name} guard words changed"


def test_noalloc_rejects_sizes_beyond_the_limit(P):
    dev = torch.device("cuda:0")
    buf = torch.zeros(16, dtype=torch.float32, device=dev)
    with pytest.raises(P.DqganError) as ei:
        P.dqgan.topk_compress_noalloc(buf, buf, buf, (1 << 20) + 1, 5, 0.1)
    assert ei.value.status == P.dqgan.ERR_INVALID_ARG and "without allocation" in str(ei.value)
    with pytest.raises(P.DqganError) as ei:
        P.dqgan.topk_compress_noalloc(buf, buf, buf, 8, 9, 0.1)
    assert ei.value.status == P.dqgan.ERR_INVALID_ARG
