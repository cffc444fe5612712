"""Guard words around every caller-owned buffer the hot path touches: the
message buffer (written by the compress kernels, read by the server), the
gradients (read only) and the parameters (read and written).  Each buffer is
a view into a larger allocation whose bytes before and after it hold a
pattern; after compress and server steps of every compressor and server
kernel family -- ragged sizes, so that every kernel's tail path runs -- the
pattern must be intact and the results must still match the oracle."""
from __future__ import annotations

import numpy as np
import pytest

import oracle
from parity_helpers import assert_messages_equal, assert_params_equal

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

LEAD = 4096   # bytes before each buffer (a multiple of 256: the views keep their alignment)
TRAIL = 4096  # bytes after it
PATTERN = 0xA5


@pytest.fixture(scope="module")
def P():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2010_13359_gb300 as P
    return P


def guarded(nbytes, dev):
    buf = torch.full((LEAD + nbytes + TRAIL,), PATTERN, dtype=torch.uint8, device=dev)
    return buf, buf[LEAD:LEAD + nbytes]


def intact(buf, nbytes):
    host = buf.cpu().numpy()
    return bool((host[:LEAD] == PATTERN).all() and (host[LEAD + nbytes:] == PATTERN).all())


CASES = [
    ("sign512", dict(d=20_011, M=5, compressor=oracle.SIGN, bucket=512)),
    ("sign4096", dict(d=(1 << 20) + 37, M=8, compressor=oracle.SIGN, bucket=4096)),
    ("sign1024_many", dict(d=70_001, M=40, compressor=oracle.SIGN, bucket=1024)),
    ("sign64", dict(d=3_333, M=3, compressor=oracle.SIGN, bucket=64)),
    ("squant_b2", dict(d=123_457, M=16, compressor=oracle.SQUANT, bucket=512, bits=2)),
    ("squant_b4", dict(d=123_457, M=12, compressor=oracle.SQUANT, bucket=512, bits=4)),
    ("squant_b8", dict(d=123_457, M=33, compressor=oracle.SQUANT, bucket=256, bits=8)),
    ("qsgd_b4", dict(d=77_777, M=7, compressor=oracle.QSGD, bucket=512, bits=4)),
    ("identity", dict(d=10_007, M=6, compressor=oracle.IDENTITY)),
    ("topk", dict(d=300_007, M=8, compressor=oracle.TOPK, k=3_001)),
    ("topk_all", dict(d=4_099, M=3, compressor=oracle.TOPK, k=4_099)),
    ("topk_many", dict(d=20_000, M=70, compressor=oracle.TOPK, k=200)),
]


@pytest.mark.parametrize("name,kw", CASES, ids=[c[0] for c in CASES])
def test_guard_words_stay_intact(P, name, kw):
    dev = torch.device("cuda:0")
    stream = torch.cuda.current_stream(dev)
    ocfg = oracle.Config(lr=1e-2, seed=6, **kw)
    d, M = ocfg.d, ocfg.M
    h = P.create(P.make_config(d=d, M=M, compressor=ocfg.compressor, lr=ocfg.lr, bucket=ocfg.bucket, k=ocfg.k,
                               bits=ocfg.bits, seed=ocfg.seed, cuda_stream=stream.cuda_stream))
    mb = h.message_bytes()
    ld = (d + 3) // 4 * 4
    g_buf, g_view = guarded(M * ld * 4, dev)
    m_buf, m_view = guarded(M * mb, dev)
    w_buf, w_view = guarded(d * 4, dev)
    g = g_view.view(torch.float32).view(M, ld)
    msgs = m_view.view(M, mb)
    w = w_view.view(torch.float32)
    rng = np.random.default_rng(3)
    w0 = (rng.standard_normal(d) * 0.02).astype(np.float32)
    w.copy_(torch.from_numpy(w0))
    st = oracle.State(ocfg)
    w_orc = w0.copy()
    for t in range(2):
        gh = (rng.standard_normal((M, d)) * np.exp(rng.uniform(-3, 1, (M, d)))).astype(np.float32)
        g[:, :d].copy_(torch.from_numpy(gh))
        h.workers_compress_all(g, ld, msgs)
        h.server_aggregate_update(msgs, w)
        h.synchronize()
        want = st.step(gh, w_orc)
        got = msgs.cpu().numpy()
        for i in range(M):
            assert_messages_equal(ocfg, got[i], want[i], f"{name} worker {i} step {t}")
        assert_params_equal(w.cpu().numpy(), w_orc, f"{name} step {t}")
        for label, buf, n in (("gradients", g_buf, M * ld * 4), ("messages", m_buf, M * mb), ("params", w_buf, d * 4)):
            assert intact(buf, n), f"{name} step {t}: guard words around the {label} changed"
    h.destroy()
