"""Golden fixture: three steps of Algorithm 2 on a tiny dyadic problem for
each compressor (tests/golden/algorithm2_tiny.json, written by
tests/golden/make_golden.py from the oracle after checking it against the
exact rational replay).  The CPU test pins the oracle to the stored bytes;
the GPU test runs the CUDA path on the same inputs against them."""
from __future__ import annotations

import json
import os

import numpy as np
import pytest

import oracle

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "algorithm2_tiny.json")


def load():
    with open(GOLDEN) as f:
        data = json.load(f)
    T, M, D = data["steps"], data["M"], data["d"]
    g = np.array([[[int(x, 16) for x in row] for row in step] for step in data["gradients_f32_hex"]],
                 dtype=np.uint32).view(np.float32).reshape(T, M, D)
    w0 = np.array([int(x, 16) for x in data["w0_f32_hex"]], dtype=np.uint32).view(np.float32)
    return data, g, w0


def f32(hexes):
    return np.array([int(x, 16) for x in hexes], dtype=np.uint32).view(np.float32)


CASE_NAMES = ["sign", "topk", "squant_b4", "identity"]


@pytest.mark.parametrize("name", CASE_NAMES)
def test_oracle_reproduces_golden(name):
    data, g, w0 = load()
    case = data["cases"][name]
    cfg = oracle.Config(d=data["d"], M=data["M"], lr=data["lr"], seed=data["seed"], **case["config"])
    st = oracle.State(cfg)
    w = w0.copy()
    for t, want in enumerate(case["steps"]):
        msgs = st.step(g[t], w)
        for m in range(data["M"]):
            assert msgs[m].tobytes().hex() == want["messages_hex"][m], (name, t, m)
            assert np.array_equal(st.e[m].view(np.uint32), f32(want["e_f32_hex"][m]).view(np.uint32))
        assert np.array_equal(w.view(np.uint32), f32(want["w_f32_hex"]).view(np.uint32))


@pytest.mark.gpu
@pytest.mark.parametrize("name", CASE_NAMES)
def test_cuda_path_reproduces_golden(name):
    torch = pytest.importorskip("torch")
    import __graft_entry__
    __graft_entry__.build()
    import paper_2010_13359_gb300 as P
    data, g, w0 = load()
    case = data["cases"][name]
    kw = dict(case["config"])
    D, M = data["d"], data["M"]
    dev = torch.device("cuda:0")
    stream = torch.cuda.current_stream(dev)
    h = P.create(P.make_config(d=D, M=M, lr=data["lr"], seed=data["seed"], cuda_stream=stream.cuda_stream,
                               compressor=kw.pop("compressor"), **kw))
    mb = h.message_bytes()
    ld = (D + 3) // 4 * 4
    w = torch.from_numpy(w0.copy()).to(dev)
    msgs = torch.zeros((M, mb), dtype=torch.uint8, device=dev)
    for t, want in enumerate(case["steps"]):
        gd = torch.zeros((M, ld), dtype=torch.float32, device=dev)
        gd[:, :D] = torch.from_numpy(g[t]).to(dev)
        h.workers_compress_all(gd, ld, msgs)
        h.server_aggregate_update(msgs, w)
        got = msgs.cpu().numpy()
        for m in range(M):
            assert got[m].tobytes().hex() == want["messages_hex"][m], (name, t, m)
            e = np.empty(D, np.float32)
            h.get_residual(m, e)
            assert np.array_equal(e.view(np.uint32), f32(want["e_f32_hex"][m]).view(np.uint32))
        w_want = f32(want["w_f32_hex"])
        assert np.array_equal(w.cpu().numpy().view(np.uint32), w_want.view(np.uint32)), (name, t, "params")
    h.destroy()
