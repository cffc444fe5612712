"""Per-layer bucketing (dqgan_set_segments) against the oracle: buckets
restart at every layer boundary, so the scale sections grow by the partial
buckets and every scale covers exactly its own bucket.  Messages, residuals
and lookahead offsets bit for bit, parameters within the step tolerance,
over several free-running steps; plus the call's argument rules."""
from __future__ import annotations

import numpy as np
import pytest

import oracle
from parity_helpers import STEP_RTOL, assert_bits_equal, assert_messages_equal, oracle_config, assert_params_equal
from paper_2010_13359_gb300.workloads import WORKLOADS

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def P():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2010_13359_gb300 as P
    return P


def random_segments(rng, d, n):
    cuts = np.sort(rng.choice(np.arange(1, d // 32), size=n - 1, replace=False)) * 32
    return tuple([0, *cuts.tolist(), d])


def run_segmented(P, ocfg, T, seed):
    dev = torch.device("cuda:0")
    stream = torch.cuda.current_stream(dev)
    rng = np.random.default_rng(seed)
    h = P.create(P.make_config(d=ocfg.d, M=ocfg.M, compressor=ocfg.compressor, lr=ocfg.lr, bucket=ocfg.bucket,
                               bits=ocfg.bits, seed=ocfg.seed, flags=P.KEEP_LOOKAHEAD if ocfg.keep_lookahead else 0,
                               cuda_stream=stream.cuda_stream))
    h.set_segments(ocfg.segments)
    assert h.message_bytes() == oracle.message_bytes(ocfg)
    st = oracle.State(ocfg)
    d, M = ocfg.d, ocfg.M
    ld = (d + 3) // 4 * 4
    w0 = (rng.standard_normal(d) * 0.02).astype(np.float32)
    w_gpu = torch.from_numpy(w0.copy()).to(dev)
    w_orc = w0.copy()
    msgs = torch.zeros((M, h.message_bytes()), dtype=torch.uint8, device=dev)
    for t in range(1, T + 1):
        g = (rng.standard_normal((M, d)) * np.exp(rng.uniform(-4, 1, (M, d)))).astype(np.float32)
        g_dev = torch.zeros((M, ld), dtype=torch.float32, device=dev)
        g_dev[:, :d] = torch.from_numpy(g).to(dev)
        h.workers_compress_all(g_dev, ld, msgs)
        want = st.compress_all(g)
        got = msgs.cpu().numpy()
        for i in range(M):
            assert_messages_equal(ocfg, got[i], want[i], f"worker {i} step {t}")
            e_i = np.empty(d, np.float32)
            h.get_residual(i, e_i)
            assert_bits_equal(e_i, st.e[i], f"residual worker {i} step {t}")
            if ocfg.keep_lookahead:
                h_i = np.empty(d, np.float32)
                h.get_lookahead(i, h_i)
                assert_bits_equal(h_i, st.h[i], f"lookahead offset worker {i} step {t}")
        h.server_aggregate_update(msgs, w_gpu)
        st.server(want, w_orc)
        h.synchronize()
        assert_params_equal(w_gpu.cpu().numpy(), w_orc, "params")
    h.destroy()


CASES = [
    (oracle.SIGN, dict(bucket=256)), (oracle.SIGN, dict(bucket=1024)), (oracle.SIGN, dict(bucket=4096)),
    (oracle.SQUANT, dict(bucket=512, bits=2)), (oracle.SQUANT, dict(bucket=512, bits=4)),
    (oracle.SQUANT, dict(bucket=2048, bits=8)), (oracle.QSGD, dict(bucket=1024, bits=8)),
]


def _id(case):
    comp, kw = case
    return {0: "sign", 2: "squant", 4: "qsgd"}[comp] + "-" + "-".join(f"{k}{v}" for k, v in kw.items())


@pytest.mark.parametrize("case", CASES, ids=_id)
@pytest.mark.parametrize("layout", ["random7", "tiny_and_long", "one"])
def test_segmented_matches_oracle(P, case, layout):
    comp, kw = case
    d = 20_011
    if layout == "random7":
        segs = random_segments(np.random.default_rng(kw["bucket"]), d, 7)
    elif layout == "tiny_and_long":
        segs = (0, 32, 64, 96, 5_024, 5_056, d)
    else:
        segs = (0, d)
    ocfg = oracle_config(d, 3, comp, lr=0.05, seed=77, keep=True, segments=segs, **kw)
    run_segmented(P, ocfg, T=3, seed=len(segs))


@pytest.mark.parametrize("comp", [oracle.SQUANT, oracle.QSGD], ids=["squant", "qsgd"])
@pytest.mark.parametrize("layout", ["random7", "tiny_and_long", "one", "odd_words"])
def test_segmented_8bit_sixteen_workers(P, comp, layout):
    """8-bit codes with 16 workers take the server whose slices come from the
    per-bucket table (no slice spans two buckets; short slices at the end of
    a layer's last bucket store only their own rows)."""
    d = 40_011
    if layout == "random7":
        segs = random_segments(np.random.default_rng(11), d, 7)
    elif layout == "tiny_and_long":
        segs = (0, 32, 64, 96, 5_024, 5_056, d)
    elif layout == "odd_words":  # layer starts on every residue of 4 code words
        segs = (0, 96, 224, 384, 544, 9_600, 9_632, d)
    else:
        segs = (0, d)
    ocfg = oracle_config(d, 16, comp, lr=0.05, seed=5, keep=False, segments=segs, bucket=512, bits=8)
    run_segmented(P, ocfg, T=3, seed=len(segs) + 16)


@pytest.mark.parametrize("name", ["dcgan_sign_layers", "resnet_squant_b8_layers"])
def test_layer_workloads_first_steps(P, name):
    """The per-layer workloads at a reduced size: their own 16 / 64 layer
    segments scaled to d = 2^20, M = 4, three free-running steps."""
    wl = WORKLOADS[name]
    sizes, _ = wl.segments()
    scale = (1 << 20) / wl.d
    offs = [0]
    for s in sizes[:-1]:
        offs.append(offs[-1] + max(32, int(s * scale) // 32 * 32))
    offs = [o for o in offs if o < (1 << 20)] + [1 << 20]
    ocfg = oracle_config(1 << 20, 4, wl.compressor, lr=wl.lr, bucket=wl.bucket, bits=wl.bits, seed=wl.seed,
                         segments=tuple(offs))
    run_segmented(P, ocfg, T=3, seed=5)


def test_set_segments_argument_rules(P):
    dev = torch.device("cuda:0")
    d = 4_096
    h = P.create(P.make_config(d=d, M=2, compressor=P.SIGN, bucket=512))
    flat = h.message_bytes()
    for bad in [(0, 100, d), (0, 64, 64, d), (32, d), (0, 64, d + 32), (0, 2048, 1024, d)]:
        with pytest.raises(P.DqganError) as exc:
            h.set_segments(bad)
        assert exc.value.status == P.dqgan.ERR_INVALID_ARG
    assert h.message_bytes() == flat
    h.set_segments((0, 96, d))
    seg_cfg = oracle_config(d, 2, oracle.SIGN, bucket=512, segments=(0, 96, d))
    assert h.message_bytes() == oracle.message_bytes(seg_cfg)
    h.set_segments(None)
    assert h.message_bytes() == flat
    g = torch.zeros((2, d), dtype=torch.float32, device=dev)
    msgs = torch.zeros((2, flat), dtype=torch.uint8, device=dev)
    w = torch.zeros(d, dtype=torch.float32, device=dev)
    h.workers_compress_all(g, d, msgs)
    h.server_aggregate_update(msgs, w)
    with pytest.raises(P.DqganError) as exc:
        h.set_segments((0, 96, d))
    assert exc.value.status == P.dqgan.ERR_INVALID_ARG and "before the first step" in str(exc.value)
    h.destroy()
    t = P.create(P.make_config(d=d, M=2, compressor=P.TOPK, k=10))
    with pytest.raises(P.DqganError) as exc:
        t.set_segments((0, 96, d))
    assert exc.value.status == P.dqgan.ERR_UNSUPPORTED
    t.destroy()
