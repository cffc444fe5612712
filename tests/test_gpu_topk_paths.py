"""The top-k worker step's two routes to the same result, against the oracle.

The first pass writes, per tile, the elements whose top key digit reaches a
threshold carried over from the worker's previous call; the second kernel
uses them when the new top digit of the k-th largest key is not below that
threshold, and otherwise re-extracts the candidates from p.  Whichever route
a call takes, the records and residuals must be the oracle's bit for bit:

* a scale sequence that makes the threshold fall (re-extraction), rise far
  (many candidates), land inside big groups of equal keys, and sit on an
  all-zero p;
* more candidates than a select CTA keeps on chip (k = d/2);
* server paths for up to 64 workers (per-index worker masks, one owner
  per index) and beyond (a thread per record);
* at d = 7e7 the CTAs' tiles no longer fit one chunk of tile counts; there
  the selection is checked by the properties that define it uniquely
  (k records in index order holding p_j, no dropped key above the smallest
  kept key, equal keys kept lowest index first, e = +0 exactly there).
"""
from __future__ import annotations

import numpy as np
import pytest

import oracle
from parity_helpers import assert_bits_equal, assert_messages_equal, oracle_config

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def P():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2010_13359_gb300 as P
    return P


def handle(P, ocfg, stream):
    return P.create(P.make_config(d=ocfg.d, M=ocfg.M, compressor=oracle.TOPK, lr=ocfg.lr, k=ocfg.k,
                                  seed=ocfg.seed, flags=P.KEEP_LOOKAHEAD if ocfg.keep_lookahead else 0,
                                  cuda_stream=stream.cuda_stream))


def step_grads(kind, M, d, rng):
    if kind == "ties":
        return (rng.integers(-3, 4, size=(M, d)) * 0.25).astype(np.float32)
    if kind == "zeros":
        return np.zeros((M, d), np.float32)
    return (rng.standard_normal((M, d)) * np.float32(kind)).astype(np.float32)


def run_free(P, ocfg, kinds, seed=0):
    dev = torch.device("cuda:0")
    stream = torch.cuda.current_stream(dev)
    rng = np.random.default_rng(seed)
    h = handle(P, ocfg, stream)
    st = oracle.State(ocfg)
    d, M = ocfg.d, ocfg.M
    ld = (d + 3) // 4 * 4
    msgs = torch.zeros((M, h.message_bytes()), dtype=torch.uint8, device=dev)
    w = torch.zeros(d, dtype=torch.float32, device=dev)
    w_orc = np.zeros(d, np.float32)
    for t, kind in enumerate(kinds, start=1):
        g = step_grads(kind, M, d, rng)
        g_dev = torch.zeros((M, ld), dtype=torch.float32, device=dev)
        g_dev[:, :d] = torch.from_numpy(g).to(dev)
        h.workers_compress_all(g_dev, ld, msgs)
        want = st.compress_all(g)
        got = msgs.cpu().numpy()
        for i in range(M):
            assert_messages_equal(ocfg, got[i], want[i], f"step {t} ({kind}) worker {i}")
            e_i = np.empty(d, np.float32)
            h.get_residual(i, e_i)
            assert_bits_equal(e_i, st.e[i], f"residual step {t} ({kind}) worker {i}")
            if ocfg.keep_lookahead:
                h_i = np.empty(d, np.float32)
                h.get_lookahead(i, h_i)
                assert_bits_equal(h_i, st.h[i], f"lookahead offset step {t} ({kind}) worker {i}")
        h.server_aggregate_update(msgs, w)
        st.server(want, w_orc)
    h.synchronize()
    assert np.array_equal(w.cpu().numpy().view(np.uint32), w_orc.view(np.uint32))
    h.destroy()


@pytest.mark.parametrize("d,k", [(200_003, 3_000), (40_000, 39_000), (5_000, 17)])
def test_threshold_carry_routes(P, d, k):
    kinds = [1.0, 1.0, 1e-3, 1e-3, 1e3, "ties", "ties", "zeros", 1.0, 1e-30]
    ocfg = oracle_config(d, 2, oracle.TOPK, lr=0.5, k=k, seed=3, keep=True)
    run_free(P, ocfg, kinds, seed=d)


def test_candidates_beyond_on_chip_copy(P):
    ocfg = oracle_config(1_000_003, 1, oracle.TOPK, lr=0.1, k=500_000, seed=4, keep=False)
    run_free(P, ocfg, [1.0, 1.0, 0.5], seed=1)


def test_many_tiles_per_cta_properties(P):
    dev = torch.device("cuda:0")
    stream = torch.cuda.current_stream(dev)
    d, k, lr = 70_000_001, 700_000, 0.25
    h = P.create(P.make_config(d=d, M=1, compressor=oracle.TOPK, lr=lr, k=k, cuda_stream=stream.cuda_stream))
    ld = (d + 3) // 4 * 4
    gen = torch.Generator(device=dev)
    e_prev = np.zeros(d, np.float32)
    msg = torch.zeros(h.message_bytes(), dtype=torch.uint8, device=dev)
    for t in range(1, 3):
        gen.manual_seed(100 + t)
        g = torch.randn(ld, generator=gen, device=dev, dtype=torch.float32)
        h.worker_compress(0, g, msg)
        h.synchronize()
        p = (np.float32(lr) * g[:d].cpu().numpy()).astype(np.float32) + e_prev
        rec = msg[:8 * k].cpu().numpy().view(np.uint32).reshape(k, 2)
        idx = rec[:, 0].astype(np.int64)
        assert np.all(np.diff(idx) > 0) and idx[0] >= 0 and idx[-1] < d
        assert np.array_equal(rec[:, 1], p[idx].view(np.uint32))
        key = p.view(np.uint32) & 0x7FFFFFFF
        kept = np.zeros(d, bool)
        kept[idx] = True
        T = key[idx].min()
        assert key[~kept].max(initial=0) <= T
        ties_kept = idx[key[idx] == T]
        ties_dropped = np.flatnonzero((~kept) & (key == T))
        if ties_dropped.size:
            assert ties_kept.max() < ties_dropped.min()
        e = np.empty(d, np.float32)
        h.get_residual(0, e)
        want_e = p.copy()
        want_e[idx] = np.float32(0.0)
        assert_bits_equal(e, want_e, f"residual step {t}")
        e_prev = e
        h.set_step(t + 1)
    h.destroy()


@pytest.mark.parametrize("M", [33, 64, 65, 70])
def test_server_worker_counts(P, M):
    """Up to 64 workers the server scatters into per-index worker masks and
    the lowest worker of each index sums it; above, one thread per record
    searches the other workers' records.  Both sum in the library's pairwise
    order, so w matches bit for bit."""
    ocfg = oracle_config(50_003, M, oracle.TOPK, lr=0.5, k=777, seed=M, keep=False)
    run_free(P, ocfg, [1.0, 1.0, "ties"], seed=M)
