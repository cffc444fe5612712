"""Sign server (decode + average + update, Algorithm 2) on the shapes that
select its TMA paths: buckets of 1024..4096 with M <= 32, where the message
words and the parameters are staged by TMA and each lane transposes a
32 x 32 bit block in registers.

Both kernels run on every shape, with flat buckets and with layer
segments (forced by DQGAN_SIGN_SERVER, read when a handle is created), and
once more with the choice by size.

The messages come from the GPU compress step and are checked bit for bit
against the oracle's; the oracle's server then runs on the same messages and
the parameters must agree within the step tolerance and then bit for bit
(both sum over workers in the library's pairwise order).  Parameters past d must
stay untouched: the vector sits inside a larger buffer whose tail holds
sentinels.  Sizes cover d < 32 (no parameter map), d a multiple of 32, a
partial last row, a partial row that starts a slice of its own (floor(d/32)
a multiple of 32), ragged last buckets and one full-size-like case.
"""
from __future__ import annotations

import numpy as np
import pytest

import oracle
from parity_helpers import STEP_RTOL, assert_messages_equal, oracle_config, assert_params_equal

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def P():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2010_13359_gb300 as P
    return P


CASES = [
    # (d, M, bucket)
    (7, 4, 1024),                # below one row: per-element fallback
    (32, 1, 1024),               # one full row
    (33, 5, 1024),               # one row and a partial one
    (1023, 8, 1024),             # one partial bucket
    (32 * 32 * 3 + 5, 13, 1024),  # the partial row begins a slice
    (4096 * 7 + 31, 31, 4096),   # M = 31: the seventh group holds one worker
    (4096 * 7 + 31, 32, 4096),
    (2048 * 9 + 64, 32, 2048),
    (200_003, 16, 2048),
    (1 << 20, 32, 4096),
    (1_000_037, 8, 1024),
    (1_000_037, 30, 4096),       # NG = 6
    (9_000_011, 8, 4096),        # large enough for the column kernel by size
]


@pytest.mark.parametrize("path", ["col", "tma", "auto"])
@pytest.mark.parametrize("d,M,bucket", CASES, ids=[f"d{d}-M{M}-b{b}" for d, M, b in CASES])
def test_sign_server_paths(P, d, M, bucket, path, monkeypatch):
    """Each kernel forced through DQGAN_SIGN_SERVER, and the choice by size."""
    dev = torch.device("cuda:0")
    stream = torch.cuda.current_stream(dev)
    ocfg = oracle_config(d, M, oracle.SIGN, lr=0.03, bucket=bucket, seed=d + M)
    if path == "auto":
        monkeypatch.delenv("DQGAN_SIGN_SERVER", raising=False)
    else:
        monkeypatch.setenv("DQGAN_SIGN_SERVER", path)
    h = P.create(P.make_config(d=d, M=M, compressor=P.SIGN, lr=0.03, bucket=bucket, seed=d + M,
                               cuda_stream=stream.cuda_stream))
    rng = np.random.default_rng(d * 7 + M)
    st = oracle.State(ocfg)
    ld = (d + 3) // 4 * 4
    guard = 64
    w0 = (rng.standard_normal(d) * 0.02).astype(np.float32)
    buf = torch.full((d + guard,), 12345.0, dtype=torch.float32, device=dev)
    buf[:d] = torch.from_numpy(w0).to(dev)
    w_gpu = buf[:d]
    w_orc = w0.copy()
    # two parameter buffers in turn: the cached TMA map follows the pointer
    alt = torch.zeros(d + guard, dtype=torch.float32, device=dev)
    mb = h.message_bytes()
    for t in range(3):
        g = (rng.standard_normal((M, d)) * np.exp(rng.uniform(-3, 1, (M, d)))).astype(np.float32)
        g_dev = torch.zeros((M, ld), dtype=torch.float32, device=dev)
        g_dev[:, :d] = torch.from_numpy(g).to(dev)
        msgs = torch.zeros((M, mb), dtype=torch.uint8, device=dev)
        h.workers_compress_all(g_dev, ld, msgs)
        msgs_orc = st.compress_all(g)
        got = msgs.cpu().numpy()
        for i in range(M):
            assert_messages_equal(ocfg, got[i], msgs_orc[i], f"worker {i} step {t}")
        if t == 1:  # this step runs on the other buffer
            alt[:d] = w_gpu
            h.server_aggregate_update(msgs, alt[:d])
            w_gpu.copy_(alt[:d])
        else:
            h.server_aggregate_update(msgs, w_gpu)
        st.server(msgs_orc, w_orc)
        h.synchronize()
        assert_params_equal(w_gpu.cpu().numpy(), w_orc, f"step {t}")
    tail = buf[d:].cpu().numpy()
    assert np.all(tail == 12345.0), "parameters past d were written"
    assert torch.all(alt[d:] == 0.0)
    h.destroy()


def layer_offsets(kind, d, rng):
    if kind == "tiny":  # many one-word layers, then a long one
        return tuple([0, *range(32, 32 * 40, 32), d])
    if kind == "odd":  # layer sizes that leave every bucket off the 16-byte grid of the payload
        offs, at = [0], 0
        while True:
            at += 32 * int(rng.integers(1, 90))
            if at >= d:
                break
            offs.append(at)
        return tuple(offs + [d])
    cuts = np.sort(rng.choice(np.arange(1, d // 32), size=15, replace=False)) * 32
    return tuple([0, *cuts.tolist(), d])


SEG_CASES = [
    (20_011, 3, 1024, "tiny"), (65_536, 8, 1024, "odd"), (65_536 + 7, 32, 4096, "odd"),
    (200_003, 13, 2048, "random16"), (2_000_000, 8, 1024, "random16"), (1_000_003, 31, 4096, "random16"),
]


@pytest.mark.parametrize("path", ["col", "tma", "auto"])
@pytest.mark.parametrize("d,M,bucket,kind", SEG_CASES, ids=[f"d{d}-M{M}-b{b}-{k}" for d, M, b, k in SEG_CASES])
def test_sign_server_segments(P, d, M, bucket, kind, path, monkeypatch):
    """Layer segments, both kernels (forced, and chosen by size): every slice
    lies inside one bucket; the column kernel updates short slices with
    plain stores, the warp-transpose kernel realigns each slice's words in
    its box and stores only the slice's own rows."""
    if path == "auto":
        monkeypatch.delenv("DQGAN_SIGN_SERVER", raising=False)
    else:
        monkeypatch.setenv("DQGAN_SIGN_SERVER", path)
    dev = torch.device("cuda:0")
    stream = torch.cuda.current_stream(dev)
    rng = np.random.default_rng(d + bucket)
    segs = layer_offsets(kind, d, rng)
    ocfg = oracle_config(d, M, oracle.SIGN, lr=0.03, bucket=bucket, seed=M, segments=segs)
    h = P.create(P.make_config(d=d, M=M, compressor=P.SIGN, lr=0.03, bucket=bucket, seed=M,
                               cuda_stream=stream.cuda_stream))
    h.set_segments(segs)
    st = oracle.State(ocfg)
    ld = (d + 3) // 4 * 4
    guard = 64
    w0 = (rng.standard_normal(d) * 0.02).astype(np.float32)
    buf = torch.full((d + guard,), -777.0, dtype=torch.float32, device=dev)
    buf[:d] = torch.from_numpy(w0).to(dev)
    w_gpu = buf[:d]
    w_orc = w0.copy()
    msgs = torch.zeros((M, h.message_bytes()), dtype=torch.uint8, device=dev)
    for t in range(2):
        g = (rng.standard_normal((M, d)) * np.exp(rng.uniform(-3, 1, (M, d)))).astype(np.float32)
        g_dev = torch.zeros((M, ld), dtype=torch.float32, device=dev)
        g_dev[:, :d] = torch.from_numpy(g).to(dev)
        h.workers_compress_all(g_dev, ld, msgs)
        want = st.compress_all(g)
        got = msgs.cpu().numpy()
        for i in range(M):
            assert_messages_equal(ocfg, got[i], want[i], f"worker {i} step {t}")
        h.server_aggregate_update(msgs, w_gpu)
        st.server(want, w_orc)
        h.synchronize()
        assert_params_equal(w_gpu.cpu().numpy(), w_orc, f"step {t}")
    assert np.all(buf[d:].cpu().numpy() == -777.0), "parameters past d were written"
    h.destroy()
