"""Property tests of the CPU oracle on arbitrary inputs (hypothesis).

The fixed-case pins in test_oracle_pins.py check the oracle against the
paper's identities and brute force. These tests draw many more inputs,
including heavy ties, zeros of both signs and ragged last buckets. For each
input they check what the definitions fix, by an independent route:

* top-k (Section 2.4, Theorem 1): the kept set is the first k of the indices
  sorted by (|p| descending, index ascending). The records are in ascending
  index order and carry p_j. The residual is +0 at a kept index and p_j
  elsewhere, and ||Q(p) - p||^2 <= (1 - k/d) ||p||^2;
* scaled sign (Section 2.4): in each bucket |Q_j| is one scale s_b, within
  the fp32 summation bound of mean |p_j| (computed in float64). Q_j < 0
  exactly where p_j < 0, and e = fl(p - Q);
* b-bit stochastic quantiser (Hou et al., proof of Theorem 2): s_b = max
  |p_j| of the bucket. Q_j is 0 or has the sign of p_j, |Q_j| <= s_b, and
  |Q_j - p_j| <= s_b / K (one level step), up to rounding. e = fl(p - Q);
* QSGD's variant (Eq. (qsgd)): s_b = ||p_b||_2 within the fp32 bound, the
  same sign and one-step properties;
* server (Algorithm 2): w_new = w - (1/M) sum_m Q_m, within the rounding of
  an M-term fp32 sum (float64 reference).

The tests touch no CUDA code.
"""
from __future__ import annotations

import numpy as np
import pytest

hyp = pytest.importorskip("hypothesis")
from hypothesis import given, settings, strategies as st  # noqa: E402

import oracle  # noqa: E402

U = 2.0 ** -24  # unit roundoff of binary32

# values with many exact ties (a small alphabet, both signs, both zeros) or
# spread over several binades
_ALPHABET = [0.0, -0.0, 0.5, -0.5, 1.0, -1.0, 0.25, 3.0, -3.0, 1e-3, -1e-3, 7.5]


@st.composite
def vectors(draw, max_d=160):
    d = draw(st.integers(min_value=1, max_value=max_d))
    if draw(st.booleans()):
        vals = draw(st.lists(st.sampled_from(_ALPHABET), min_size=d, max_size=d))
        x = np.array(vals, dtype=np.float32)
    else:
        seed = draw(st.integers(min_value=0, max_value=2**31 - 1))
        r = np.random.default_rng(seed)
        x = (r.standard_normal(d) * np.exp(r.uniform(-6, 2, d))).astype(np.float32)
    return x


def run_worker(cfg: oracle.Config, p: np.ndarray):
    """One oracle worker step with g = p, lr = 1 and e = 0, so that p is the
    error-compensated vector up to the sign of zero (fl(g + 0) turns -0 into +0)."""
    e = np.zeros(cfg.d, dtype=np.float32)
    msg = oracle.worker_step(cfg, 0, 1, p, e)
    p_formed = (np.float32(1.0) * p + np.float32(0.0)).astype(np.float32)
    return p_formed, msg, e


def key(x: np.ndarray) -> np.ndarray:
    return x.view(np.uint32) & np.uint32(0x7FFFFFFF)


SETTINGS = settings(max_examples=60, deadline=None)


@SETTINGS
@given(x=vectors(), kfrac=st.floats(min_value=0.0, max_value=1.0))
def test_topk_keeps_the_k_largest_with_lower_index_ties(x, kfrac):
    d = x.size
    k = max(1, min(d, int(round(kfrac * d))))
    cfg = oracle.Config(d=d, M=1, compressor=oracle.TOPK, lr=1.0, k=k)
    p, msg, e = run_worker(cfg, x)
    order = sorted(range(d), key=lambda j: (-int(key(p[j:j + 1])[0]), j))
    want = np.zeros(d, dtype=bool)
    want[order[:k]] = True
    assert np.array_equal(oracle.topk_select(p, k), want)
    rec = msg[:8 * k].view(np.uint32).reshape(k, 2)
    idx = rec[:, 0].astype(np.int64)
    assert np.all(np.diff(idx) > 0) and np.array_equal(np.flatnonzero(want), idx)
    assert np.array_equal(rec[:, 1], p[idx].view(np.uint32))
    e_want = np.where(want, np.float32(0.0), p).astype(np.float32)
    assert np.array_equal(e.view(np.uint32), e_want.view(np.uint32))
    q = oracle.decode(cfg, msg).astype(np.float64)
    pd = p.astype(np.float64)
    assert np.sum((q - pd) ** 2) <= (1.0 - k / d) * np.sum(pd ** 2) * (1 + 1e-12) + 1e-300


@SETTINGS
@given(x=vectors(), bucket=st.sampled_from([32, 64, 128]))
def test_sign_scales_signs_and_residual(x, bucket):
    d = x.size
    cfg = oracle.Config(d=d, M=1, compressor=oracle.SIGN, lr=1.0, bucket=bucket)
    p, msg, e = run_worker(cfg, x)
    q = oracle.decode(cfg, msg)
    for b0 in range(0, d, bucket):
        pb, qb = p[b0:b0 + bucket], q[b0:b0 + bucket]
        n = pb.size
        mags = np.abs(qb)
        assert np.all(mags == mags[0]), "one scale per bucket"
        mean_abs = np.sum(np.abs(pb.astype(np.float64))) / n
        # (n - 1) roundings of the fp32 sum, one of the division
        assert abs(float(mags[0]) - mean_abs) <= (n * U) * mean_abs + 1e-45
    assert np.array_equal(q < 0, p < 0), "Q_j < 0 exactly where p_j < 0"
    assert np.array_equal(e.view(np.uint32), (p - q).astype(np.float32).view(np.uint32))


@SETTINGS
@given(x=vectors(), bits=st.sampled_from([2, 4, 8]), bucket=st.sampled_from([32, 64]),
       seed=st.integers(min_value=0, max_value=2**32 - 1))
def test_squant_levels_are_within_one_step(x, bits, bucket, seed):
    d = x.size
    K = (1 << (bits - 1)) - 1
    cfg = oracle.Config(d=d, M=1, compressor=oracle.SQUANT, lr=1.0, bucket=bucket, bits=bits, seed=seed)
    p, msg, e = run_worker(cfg, x)
    q = oracle.decode(cfg, msg)
    off_s = oracle.layout(cfg)[0]
    nb = -(-d // bucket)
    scales = msg[off_s:off_s + 4 * nb].view(np.float32)
    for b in range(nb):
        pb = p[b * bucket:(b + 1) * bucket].astype(np.float64)
        qb = q[b * bucket:(b + 1) * bucket].astype(np.float64)
        s = float(np.max(np.abs(pb)))
        assert float(scales[b]) == s, "the l_inf scale is the exact max"
        assert np.all(np.abs(qb) <= s * (1 + 2 * U))
        assert np.all((qb == 0) | (np.sign(qb) == np.sign(pb)))
        assert np.all(np.abs(qb - pb) <= s / K * (1 + 4 * U) + 2 * U * s)
    assert np.array_equal(e.view(np.uint32), (p - q).astype(np.float32).view(np.uint32))


@SETTINGS
@given(M=st.integers(min_value=1, max_value=6), x=vectors(max_d=96),
       comp=st.sampled_from([oracle.SIGN, oracle.SQUANT, oracle.IDENTITY]),
       seed=st.integers(min_value=0, max_value=1000))
def test_server_subtracts_the_average(M, x, comp, seed):
    d = x.size
    cfg = oracle.Config(d=d, M=M, compressor=comp, lr=1.0, bucket=32, bits=4, seed=seed)
    r = np.random.default_rng(seed)
    g = (x[None, :] * r.uniform(0.5, 2.0, (M, 1))).astype(np.float32)
    st_ = oracle.State(cfg)
    msgs = st_.compress_all(g)
    w0 = (r.standard_normal(d) * 0.02).astype(np.float32)
    w = w0.copy()
    st_.server(msgs, w)
    qs = np.stack([oracle.decode(cfg, msgs[m]) for m in range(M)]).astype(np.float64)
    avg = qs.sum(axis=0) / M
    bound = (M + 1) * U * np.sum(np.abs(qs), axis=0) / M + U * np.abs(w0.astype(np.float64) - avg)
    assert np.all(np.abs(w.astype(np.float64) - (w0.astype(np.float64) - avg)) <= bound + 1e-45)


@SETTINGS
@given(x=vectors(), bits=st.sampled_from([2, 4, 8]), bucket=st.sampled_from([32, 64]),
       seed=st.integers(min_value=0, max_value=2**32 - 1))
def test_qsgd_scale_is_the_l2_norm_and_levels_step_by_s_over_K(x, bits, bucket, seed):
    """QSGD's variant (Section 2.4, Eq. (qsgd)): s_b = ||p_b||_2 within the
    fp32 bound of an n-term sum of squares and one square root; Q_j is 0 or
    has the sign of p_j, and |Q_j - p_j| <= s_b / K up to rounding."""
    d = x.size
    K = (1 << (bits - 1)) - 1
    cfg = oracle.Config(d=d, M=1, compressor=oracle.QSGD, lr=1.0, bucket=bucket, bits=bits, seed=seed)
    p, msg, e = run_worker(cfg, x)
    q = oracle.decode(cfg, msg)
    off_s = oracle.layout(cfg)[0]
    nb = -(-d // bucket)
    scales = msg[off_s:off_s + 4 * nb].view(np.float32)
    for b in range(nb):
        pb = p[b * bucket:(b + 1) * bucket].astype(np.float64)
        qb = q[b * bucket:(b + 1) * bucket].astype(np.float64)
        n = pb.size
        l2 = float(np.sqrt(np.sum(pb * pb)))
        s = float(scales[b])
        if l2 < 1e-18:  # squares below the fp32 range flush the sum
            continue
        assert abs(s - l2) <= (n * U + 2 * U) * l2
        assert np.all((qb == 0) | (np.sign(qb) == np.sign(pb)))
        assert np.all(np.abs(qb) <= s * (1 + 2 * U))
        assert np.all(np.abs(qb - pb) <= s / K * (1 + 4 * U) + 2 * U * s)
    assert np.array_equal(e.view(np.uint32), (p - q).astype(np.float32).view(np.uint32))
