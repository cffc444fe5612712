"""The input recipe (seeded synthetic stand-ins for the paper's GAN workloads)
against what it promises: the sizes, worker counts, compressors, buckets and
run lengths of the workload table; valid layer segments; per-(step, worker)
gradient streams that are reproducible and distinct; per-segment scales; and
the heavy tails of the stress case.  CPU only (numpy generators)."""
from __future__ import annotations

import numpy as np
import pytest

from paper_2010_13359_gb300.workloads import IDENTITY, QSGD, SIGN, SQUANT, TOPK, WORKLOADS, sweep_workload


def test_workload_table_shapes():
    t = WORKLOADS["tiny_sign"]
    assert (t.d, t.M, t.compressor, t.bucket, t.steps) == (65_536, 4, SIGN, 512, 20)
    assert t.segment_offsets() == (0, 16_384, 32_768, 49_152, 65_536)
    assert t.segments()[1] == [1e-1, 3e-2, 1e-2, 3e-3]
    for name in ("dcgan_sign", "dcgan_topk", "dcgan_sign_layers"):
        w = WORKLOADS[name]
        assert (w.d, w.M, w.steps, w.n_segments) == (3_600_000, 8, 100, 16)
        assert w.std_range == (1e-4, 1e-1)
    assert WORKLOADS["dcgan_sign"].bucket == 1024 and WORKLOADS["dcgan_sign"].compressor == SIGN
    assert WORKLOADS["dcgan_topk"].compressor == TOPK and WORKLOADS["dcgan_topk"].k == 36_000  # 1 % of d
    for b in (2, 4, 8):
        w = WORKLOADS[f"resnet_squant_b{b}"]
        assert (w.d, w.M, w.compressor, w.bucket, w.bits, w.steps, w.n_segments) == \
            (25_000_000, 16, SQUANT, 512, b, 50, 64)
        assert w.std_range == (1e-5, 1e-1)
    assert WORKLOADS["resnet_qsgd_b8"].compressor == QSGD
    assert WORKLOADS["dcgan_sign_layers"].layer_buckets and WORKLOADS["resnet_squant_b8_layers"].layer_buckets
    s = WORKLOADS["stress_sign"]
    assert (s.d, s.M, s.compressor, s.bucket, s.steps, s.dist, s.dist_scale) == \
        (100_000_000, 32, SIGN, 4096, 20, "student_t3", 1e-3)
    assert IDENTITY not in {w.compressor for w in WORKLOADS.values()}


@pytest.mark.parametrize("name", sorted(WORKLOADS))
def test_segments_are_valid(name):
    w = WORKLOADS[name]
    offs = w.segment_offsets()
    sizes, stds = w.segments()
    assert offs[0] == 0 and offs[-1] == w.d and len(offs) == w.n_segments + 1
    assert all(b > a for a, b in zip(offs[:-1], offs[1:]))
    assert all(o % 32 == 0 for o in offs[1:-1]), "inner layer boundaries on 32-element words"
    assert len(stds) == w.n_segments
    lo, hi = w.std_range
    if w.segment_std is None:
        assert all(lo <= s <= hi for s in stds)
    assert w.segments() == (sizes, stds), "segment draw is seeded"


def small(name, d=1 << 16, **kw):
    return WORKLOADS[name].replace(d=d, **kw)


def test_gradient_streams_reproducible_and_distinct():
    w = small("dcgan_sign")
    a = w.gradient_np(3, 1)
    assert np.array_equal(a.view(np.uint32), w.gradient_np(3, 1).view(np.uint32))
    for step, worker in ((3, 2), (4, 1), (1, 1)):
        assert not np.array_equal(a, w.gradient_np(step, worker))
    g = w.gradients_np(2)
    assert g.shape == (w.M, w.d) and g.dtype == np.float32
    assert np.array_equal(g[5], w.gradient_np(2, 5))
    w0 = w.w0_np()
    assert w0.dtype == np.float32 and abs(float(w0.std()) - w.w0_std) < 0.05 * w.w0_std


def test_per_segment_scales():
    w = small("dcgan_sign", d=1 << 20)
    g = w.gradient_np(1, 0).astype(np.float64)
    offs = w.segment_offsets()
    _, stds = w.segments()
    for (a, b), s in zip(zip(offs[:-1], offs[1:]), stds):
        n = b - a
        est = float(np.sqrt(np.mean(g[a:b] ** 2)))
        assert abs(est - s) < 6.0 * s / np.sqrt(2 * n), (a, b, est, s)  # the sample rms within 6 sigma


def test_stress_gradients_are_heavy_tailed():
    w = small("stress_sign", d=1 << 18, segment_sizes=(1 << 18,))
    g = w.gradient_np(1, 0).astype(np.float64) / w.dist_scale
    # Student-t with 3 degrees of freedom: variance 3, and far more mass beyond
    # 6 than a normal of the same variance (whose share there is ~5e-4)
    assert abs(float(np.median(np.abs(g))) - 0.7649) < 0.02  # the t3 median of |x|
    tail = float(np.mean(np.abs(g) > 6.0))
    assert 0.0080 < tail < 0.0106, tail  # P(|t3| > 6) = 0.0093; the sample has 2^18 draws
    assert np.isfinite(g).all()


def test_sweep_sizes():
    for k in (16, 20, 27):
        w = sweep_workload(k)
        assert (w.d, w.M, w.compressor, w.bucket) == (1 << k, 8, SIGN, 1024)
        offs = w.segment_offsets()
        assert offs[-1] == w.d and all(o % 32 == 0 for o in offs[1:-1])
