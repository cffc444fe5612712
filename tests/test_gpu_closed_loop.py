"""Algorithm 2 closed around a real operator on the GPU: the lookahead feeds
the bilinear game of Section 2.2, whose operator feeds the worker step.

* Parity: with compressors whose server sums in worker order (stochastic
  quantiser, identity, top-k) the whole loop is deterministic on both sides,
  so lookahead points, messages, residuals and lookahead offsets match the
  oracle bit for bit at every step and the parameters within the step
  tolerance.  With the scaled sign the server's order differs from the
  oracle's, so the loop is checked step-locked: the oracle takes the GPU's
  parameters before each step.
* Behaviour: with the lookahead the iterates contract toward the equilibrium
  (0, 0); without it (plain simultaneous steps) they spiral outwards.
"""
from __future__ import annotations

import numpy as np
import pytest

import oracle
from parity_helpers import STEP_RTOL, assert_bits_equal, assert_messages_equal, oracle_config, assert_params_equal
from paper_2010_13359_gb300.workloads import game_diag_np, game_noise_np

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def P():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2010_13359_gb300 as P
    return P


def operator_host(w, D, noise):
    """F(x, y) = (D y, -D x) + noise, the host side of the comparison."""
    half = w.size // 2
    out = np.concatenate([D * w[half:], -(D * w[:half])]).astype(np.float32)
    return (out + noise).astype(np.float32)


def make(P, ocfg, stream):
    return P.create(P.make_config(d=ocfg.d, M=ocfg.M, compressor=ocfg.compressor, lr=ocfg.lr,
                                  bucket=ocfg.bucket, k=ocfg.k, bits=ocfg.bits, seed=ocfg.seed,
                                  flags=P.KEEP_LOOKAHEAD, cuda_stream=stream.cuda_stream))


@pytest.mark.parametrize("comp,kw,locked", [
    (oracle.SQUANT, dict(bucket=512, bits=8), False),
    (oracle.IDENTITY, dict(), False),
    (oracle.TOPK, dict(k=600), False),
    (oracle.SIGN, dict(bucket=1024), True),
])
def test_closed_loop_matches_oracle(P, comp, kw, locked):
    from paper_2010_13359_gb300.games import BilinearGame, closed_loop

    dev = torch.device("cuda:0")
    stream = torch.cuda.current_stream(dev)
    d, M, T = 8192, 4, 12
    game = BilinearGame(d=d, noise_std=0.05, seed=11)
    ocfg = oracle_config(d, M, comp, lr=0.05, seed=31, keep=True, **kw)
    h = make(P, ocfg, stream)
    st = oracle.State(ocfg)
    w0 = (np.random.default_rng(3).standard_normal(d) * 0.5).astype(np.float32)
    w_gpu = torch.from_numpy(w0.copy()).to(dev)
    w_orc = w0.copy()
    D = game_diag_np(d, game.seed)

    def on_step(t, w_half, g, msgs):
        nonlocal w_orc
        if locked:
            w_orc = w_gpu.cpu().numpy()  # the oracle starts from the GPU's parameters
        wh = w_half.cpu().numpy()
        grads = np.zeros((M, d), np.float32)
        for i in range(M):
            want_half = oracle.lookahead(w_orc, st.h[i])
            assert_bits_equal(wh[i], want_half, f"lookahead point worker {i} step {t}")
            grads[i] = operator_host(want_half, D, game_noise_np(d, game.seed, t, i, game.noise_std))
        assert_bits_equal(g[:, :d].cpu().numpy(), grads, f"operator step {t}")
        msgs_orc = st.compress_all(grads)
        got = msgs.cpu().numpy()
        for i in range(M):
            assert_messages_equal(ocfg, got[i], msgs_orc[i], f"worker {i} step {t}")
        st.server(msgs_orc, w_orc)

    for t in range(1, T + 1):
        closed_loop(h, game, w_gpu, steps=1, step0=t, on_step=on_step)
        h.synchronize()
        assert_params_equal(w_gpu.cpu().numpy(), w_orc, f"params step {t}")
        for i in range(M):
            e_i, h_i = np.empty(d, np.float32), np.empty(d, np.float32)
            h.get_residual(i, e_i)
            h.get_lookahead(i, h_i)
            assert_bits_equal(e_i, st.e[i], f"residual worker {i} step {t}")
            assert_bits_equal(h_i, st.h[i], f"lookahead offset worker {i} step {t}")
    if not locked:  # worker-order servers: the whole trajectory is exact
        assert np.array_equal(w_gpu.cpu().numpy().view(np.uint32), w_orc.view(np.uint32))
    h.destroy()


@pytest.mark.parametrize("comp,kw", [(oracle.SIGN, dict(bucket=1024)), (oracle.SQUANT, dict(bucket=512, bits=8))])
def test_lookahead_contracts_where_plain_steps_spiral(P, comp, kw):
    """Section 2.2's motivation, on the GPU through the whole compressed loop."""
    from paper_2010_13359_gb300.games import BilinearGame, closed_loop

    dev = torch.device("cuda:0")
    stream = torch.cuda.current_stream(dev)
    d, M, T = 1 << 16, 8, 300
    game = BilinearGame(d=d, noise_std=0.0, seed=5)
    ocfg = oracle_config(d, M, comp, lr=0.1, seed=2, keep=True, **kw)
    w0 = torch.from_numpy((np.random.default_rng(9).standard_normal(d)).astype(np.float32)).to(dev)
    n0 = float(w0.norm())
    assert game.d == d
    results = {}
    for look in (True, False):
        h = make(P, ocfg, stream)
        w = w0.clone()
        closed_loop(h, game, w, steps=T, lookahead=look)
        h.synchronize()
        results[look] = float(w.norm())
        h.destroy()
    # oracle runs of the same loop at d = 2^14: about 0.3 n0 with the lookahead,
    # 10x to 5000x n0 without it
    assert results[True] < 0.5 * n0
    assert results[False] > 2.0 * n0
