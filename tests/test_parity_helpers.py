"""CPU checks of the test harness itself: the oracle server run range by
range (how the full-size GPU tests and the benchmark's CPU legs split the
oracle's work over threads), or on byte-sliced sub-messages, equals the
server run once over the whole vector, with flat buckets and with layer
segments, and the per-element tolerance rule reads as stated."""
from __future__ import annotations

import numpy as np
import pytest

import oracle
from parity_helpers import rel_err, slice_messages


@pytest.mark.parametrize("comp,bits,segs", [(oracle.SIGN, 1, None), (oracle.SQUANT, 4, None),
                                            (oracle.QSGD, 2, None), (oracle.SIGN, 1, (0, 96, 1120, 5000)),
                                            (oracle.SQUANT, 8, (0, 64, 3232, 5000))])
def test_sliced_server_equals_whole(comp, bits, segs):
    d, M, bucket = 5000, 5, 256
    cfg = oracle.Config(d=d, M=M, compressor=comp, bits=bits, bucket=bucket, lr=0.01, seed=3, segments=segs)
    st = oracle.State(cfg)
    r = np.random.default_rng(4)
    msgs = st.compress_all(r.standard_normal((M, d)).astype(np.float32))
    w0 = r.standard_normal(d).astype(np.float32)
    whole = w0.copy()
    oracle.server_step(cfg, msgs, whole)
    starts = oracle.bucket_starts(cfg)
    cuts = [0, int(starts[3]), int(starts[len(starts) // 2]), int(starts[-2]), d]
    sliced = w0.copy()
    for a, b in zip(cuts[:-1], cuts[1:]):
        sub, sub_msgs = slice_messages(cfg, msgs, a, b)
        part = sliced[a:b]
        oracle.server_step(sub, sub_msgs, part)
    assert np.array_equal(sliced.view(np.uint32), whole.view(np.uint32))
    ranged = w0.copy()
    for a, b in [(0, 1), (1, 777), (777, 4099), (4099, d)]:
        oracle.server_step_range(cfg, msgs, ranged, a, b)
    assert np.array_equal(ranged.view(np.uint32), whole.view(np.uint32))


def test_rel_err_is_per_element_with_a_floor():
    y = np.array([1.0, 1e-3, 0.0, -2.0], np.float32)
    assert rel_err(y, y) == 0.0
    x = y.copy()
    x[1] = np.float32(1e-3 * (1 + 3e-5))
    assert 2.9e-5 < rel_err(x, y) < 3.1e-5           # relative to |y_j|, not to max |y|
    x = y.copy()
    x[2] = np.float32(2e-6)                           # y_j = 0: relative to 1e-6 * max |y| = 2e-6
    assert abs(rel_err(x, y) - 1.0) < 1e-6


@pytest.mark.parametrize("comp", [oracle.TOPK, oracle.IDENTITY])
def test_ranged_server_equals_whole_sparse_and_dense(comp):
    d, M = 3001, 7
    cfg = oracle.Config(d=d, M=M, compressor=comp, k=97, lr=0.5)
    st = oracle.State(cfg)
    r = np.random.default_rng(5)
    msgs = st.compress_all(r.standard_normal((M, d)).astype(np.float32))
    w0 = r.standard_normal(d).astype(np.float32)
    whole = w0.copy()
    oracle.server_step(cfg, msgs, whole)
    ranged = w0.copy()
    for a, b in [(0, 5), (5, 1000), (1000, 1001), (1001, d)]:
        oracle.server_step_range(cfg, msgs, ranged, a, b)
    assert np.array_equal(ranged.view(np.uint32), whole.view(np.uint32))
