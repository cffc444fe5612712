"""The out-of-memory paths, without exhausting the GPU: the test-only hook
DQGAN_TEST_FAIL_ALLOC=N (read by dqgan_create) makes the N-th device
allocation fail.  For every allocation that dqgan_create, dqgan_set_segments,
dqgan_set_local_workers and dqgan_set_server_optimizer make, the call must
return DQGAN_ERR_OOM, leave nothing allocated (the device's free memory is
back where it was), and -- for the calls on an existing handle -- leave the
handle usable: a step after the failure still matches the oracle."""
from __future__ import annotations

import numpy as np
import pytest

import oracle
from parity_helpers import assert_bits_equal, assert_messages_equal, assert_params_equal

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def P():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2010_13359_gb300 as P
    return P


def free_bytes():
    """Device memory free for the library: what the device reports free plus
    what torch's caching allocator holds (torch's blocks are not the
    library's, and torch may keep a segment across empty_cache)."""
    torch.cuda.synchronize()
    torch.cuda.empty_cache()
    return torch.cuda.mem_get_info()[0] + torch.cuda.memory_reserved()


def make(P, **kw):
    stream = torch.cuda.current_stream(torch.device("cuda:0"))
    return P.make_config(cuda_stream=stream.cuda_stream, **kw)


# (config, allocations dqgan_create makes): error word, e, [h], [top-k scratch]
CREATES = [
    (dict(d=1 << 20, M=4, compressor=oracle.SIGN, bucket=1024), 2),
    (dict(d=1 << 20, M=4, compressor=oracle.SIGN, bucket=1024, flags=1), 3),
    (dict(d=1 << 20, M=4, compressor=oracle.TOPK, k=1000, flags=1), 4),
]


@pytest.mark.parametrize("kw,n_alloc", CREATES, ids=["sign", "sign_lookahead", "topk_lookahead"])
def test_create_fails_cleanly_at_every_allocation(P, kw, n_alloc, monkeypatch):
    torch.zeros(1, device="cuda:0")  # context up before the first reading
    before = free_bytes()
    for n in range(1, n_alloc + 1):
        monkeypatch.setenv("DQGAN_TEST_FAIL_ALLOC", str(n))
        with pytest.raises(P.DqganError) as ei:
            P.create(make(P, **kw))
        assert ei.value.status == P.dqgan.ERR_OOM, n
        assert free_bytes() == before, f"allocation {n}: device memory leaked"
    monkeypatch.setenv("DQGAN_TEST_FAIL_ALLOC", str(n_alloc + 1))  # one past the last: create succeeds
    h = P.create(make(P, **kw))
    h.destroy()
    assert free_bytes() == before
    monkeypatch.delenv("DQGAN_TEST_FAIL_ALLOC")
    P.create(make(P, **kw)).destroy()  # disarms the hook (its count was not spent)


def step_matches_oracle(P, h, ocfg, seed):
    dev = torch.device("cuda:0")
    d, M = ocfg.d, ocfg.M
    rng = np.random.default_rng(seed)
    g = rng.standard_normal((M, d)).astype(np.float32)
    w0 = (rng.standard_normal(d) * 0.02).astype(np.float32)
    msgs = torch.zeros((M, h.message_bytes()), dtype=torch.uint8, device=dev)
    w = torch.from_numpy(w0.copy()).to(dev)
    h.workers_compress_all(torch.from_numpy(g).to(dev), d, msgs)
    h.server_aggregate_update(msgs, w)
    st = oracle.State(ocfg)
    w_orc = w0.copy()
    want = st.step(g, w_orc)
    got = msgs.cpu().numpy()
    for i in range(M):
        assert_messages_equal(ocfg, got[i], want[i], f"worker {i}")
        e = np.empty(d, np.float32)
        h.get_residual(i, e)
        assert_bits_equal(e, st.e[i], f"residual {i}")
    assert_params_equal(w.cpu().numpy(), w_orc, "params")


@pytest.mark.parametrize("what,n_calls", [("segments", 3), ("local", 1), ("optimizer", 1)])
def test_handle_calls_fail_cleanly_and_keep_the_handle(P, what, n_calls, monkeypatch):
    d, M = 1 << 20, 4
    kw = dict(d=d, M=M, compressor=oracle.SIGN, bucket=1024, lr=0.01, seed=2)
    ocfg = oracle.Config(**kw)
    segs = (0, 65536, 300_000 // 32 * 32, d)
    warm = P.create(make(P, **kw))  # the step's kernels loaded before any reading
    step_matches_oracle(P, warm, ocfg, seed=0)
    warm.destroy()
    for n in range(1, n_calls + 1):
        # create makes 2 allocations (error word, e); the n-th of the call after it fails
        monkeypatch.setenv("DQGAN_TEST_FAIL_ALLOC", str(2 + n))
        before = free_bytes()
        h = P.create(make(P, **kw))
        held = free_bytes()
        with pytest.raises(P.DqganError) as ei:
            if what == "segments":
                h.set_segments(segs)
            elif what == "local":
                h.set_local_workers(0, M)
            else:
                h.set_server_optimizer(P.dqgan.oadam(1e-3, 0.5, 0.999, 1e-8))
        assert ei.value.status == P.dqgan.ERR_OOM, (what, n)
        assert free_bytes() == held, f"{what}, allocation {n}: device memory leaked"
        step_matches_oracle(P, h, ocfg, seed=n)  # the handle is as it was
        h.destroy()
        assert free_bytes() == before
