"""Pins of the CPU oracle against what the paper and the mathematics fix.

None of these tests touches the CUDA path.  Each one would fail under a
plausible slip in the oracle (a dropped term, a wrong sign, a wrong index, a
transposed operand, a wrong tie rule):

* Definition 1 (delta-approximate compressor) and its closed form for the
  scaled sign; brute force over all sign patterns for d <= 12;
* Theorem 1 (top-k is delta = k/d) and brute force over all C(d, k) subsets;
* the moment identities in the proof of Theorem 2 (unbiasedness and the
  second moment of the b-bit stochastic quantiser), exactly by enumeration
  and statistically over Philox streams;
* the error-feedback recurrence behind Lemma 1 (per-step contraction) and the
  telescoping identity of the error-corrected sequence (Appendix B);
* Q = identity reduces Algorithm 2 to uncompressed distributed OMD, and for
  M = 1 the half-iterates obey the one-line OMD recurrence of Section 2.2;
* the fp32 oracle equals the exact-rational replay bit for bit on dyadic
  inputs, where no operation rounds;
* Philox4x32-10 against an independent implementation (Triton's, run by its
  CPU interpreter).
"""
from __future__ import annotations

import itertools
import json
import math
import os
import subprocess
import sys
from fractions import Fraction

import numpy as np
import pytest

import oracle
from oracle import exact

U32 = 2.0 ** -24  # unit roundoff of binary32


def rng(seed=0):
    return np.random.default_rng(seed)


# ---------------------------------------------------------------------------
# Philox4x32-10
# ---------------------------------------------------------------------------

TRITON_SCRIPT = r"""
import os, sys, json
os.environ["TRITON_INTERPRET"] = "1"
import torch, triton, triton.language as tl
from triton.language.random import philox_impl

@triton.jit
def kern(ctr_ptr, key_ptr, out_ptr, N: tl.constexpr):
    i = tl.arange(0, N)
    c0 = tl.load(ctr_ptr + 4 * i + 0).to(tl.uint32, bitcast=True)
    c1 = tl.load(ctr_ptr + 4 * i + 1).to(tl.uint32, bitcast=True)
    c2 = tl.load(ctr_ptr + 4 * i + 2).to(tl.uint32, bitcast=True)
    c3 = tl.load(ctr_ptr + 4 * i + 3).to(tl.uint32, bitcast=True)
    k0 = tl.load(key_ptr + 2 * i + 0).to(tl.uint32, bitcast=True)
    k1 = tl.load(key_ptr + 2 * i + 1).to(tl.uint32, bitcast=True)
    a, b, c, d = philox_impl(c0, c1, c2, c3, k0, k1, 10)
    tl.store(out_ptr + 4 * i + 0, a.to(tl.int32, bitcast=True))
    tl.store(out_ptr + 4 * i + 1, b.to(tl.int32, bitcast=True))
    tl.store(out_ptr + 4 * i + 2, c.to(tl.int32, bitcast=True))
    tl.store(out_ptr + 4 * i + 3, d.to(tl.int32, bitcast=True))

data = json.loads(sys.stdin.read())
N = len(data["ctr"])
ctr = torch.tensor(data["ctr"], dtype=torch.int64).to(torch.int32)
key = torch.tensor(data["key"], dtype=torch.int64).to(torch.int32)
out = torch.zeros(N * 4, dtype=torch.int32)
kern[(1,)](ctr.flatten(), key.flatten(), out, N)
print(json.dumps([x & 0xFFFFFFFF for x in out.tolist()]))
"""


def test_philox_matches_independent_implementation():
    """Philox4x32-10 (Salmon et al., SC'11) against Triton's own implementation."""
    pytest.importorskip("triton")
    r = rng(1)
    N = 16
    ctr = r.integers(0, 2 ** 32, size=(N, 4), dtype=np.uint64)
    key = r.integers(0, 2 ** 32, size=(N, 2), dtype=np.uint64)
    ctr[0] = 0
    key[0] = 0
    ctr[1] = 0xFFFFFFFF
    key[1] = 0xFFFFFFFF
    # torch int32 from values >= 2^31 must be wrapped first
    wrap = lambda a: [[int(v) - (1 << 32) if v >= (1 << 31) else int(v) for v in row] for row in a]
    payload = json.dumps({"ctr": wrap(ctr), "key": wrap(key)})
    env = dict(os.environ, TRITON_INTERPRET="1")
    res = subprocess.run([sys.executable, "-c", TRITON_SCRIPT], input=payload, capture_output=True,
                         text=True, env=env, timeout=300)
    if res.returncode != 0:
        pytest.skip("triton interpreter unavailable: " + res.stderr[-300:])
    theirs = np.array(json.loads(res.stdout.strip().splitlines()[-1]), dtype=np.uint64).reshape(N, 4)
    for n in range(N):
        ours = oracle.philox4x32_10(ctr[n], key[n])
        assert list(ours) == list(theirs[n]), (n, ours, theirs[n])


def test_squant_uniform_is_24_bit_and_counter_indexed():
    seed = 0x1234_5678_9ABC_DEF0
    us = [oracle.squant_uniform(seed, 3, 7, j) for j in range(64)]
    for j, u in enumerate(us):
        assert 0.0 <= u < 1.0
        assert float(u * 2 ** 24).is_integer()
        # element j uses output word j mod 4 of counter (j div 4, worker, step, 0x51)
        words = oracle.philox4x32_10([j >> 2, 3, 7, 0x51], [seed & 0xFFFFFFFF, seed >> 32])
        assert u == float(int(words[j & 3]) >> 8) * 2.0 ** -24
    # the stream depends on worker and step
    assert oracle.squant_uniform(seed, 4, 7, 0) != us[0]
    assert oracle.squant_uniform(seed, 3, 8, 0) != us[0]
    # uniformity: mean and variance of 40k draws
    draws = np.array([oracle.squant_uniform(seed, 0, 1, j) for j in range(40_000)])
    assert abs(draws.mean() - 0.5) < 5 * math.sqrt(1 / 12 / draws.size)
    assert abs(draws.var() - 1 / 12) < 0.005


# ---------------------------------------------------------------------------
# scaled sign
# ---------------------------------------------------------------------------

def sign_cfg(d, bucket, M=1, lr=1.0, keep=False):
    return oracle.Config(d=d, M=M, compressor=oracle.SIGN, lr=lr, bucket=bucket, keep_lookahead=keep)


@pytest.mark.parametrize("bucket", [32, 64, 128, 512, 1024, 4096])
@pytest.mark.parametrize("count_frac", [1.0, 0.37, 1 / 32])
def test_sign_l1_is_the_l1_norm(bucket, count_frac):
    """The fixed-order l1 sum equals the exact l1 norm within (n-1) u ||x||_1."""
    count = max(1, int(bucket * count_frac))
    x = (rng(bucket + count).standard_normal(count) * np.exp(rng(count).uniform(-8, 3, count)))
    x = x.astype(np.float32)
    got = Fraction(oracle.sign_l1(x, bucket))
    want = exact.l1(exact.frac_vec(x))
    assert abs(got - want) <= Fraction(count) * Fraction(U32) * want * Fraction(11, 10)
    # every element is counted: bumping any one element moves the sum
    for j in [0, count // 2, count - 1]:
        y = x.copy()
        y[j] = np.float32(1e6)
        assert oracle.sign_l1(y, bucket) >= 1e6


def test_sign_scale_is_mean_absolute_value_of_real_count():
    x = np.arange(1, 6, dtype=np.float32)  # a partial bucket of 5 in a bucket of 32
    assert oracle.sign_scale(x, 32) == np.float32(15.0) / np.float32(5.0)
    assert oracle.sign_scale(np.zeros(7, np.float32), 32) == 0.0


def test_sign_message_layout_and_residual():
    """Bits: 1 iff p < 0, little-endian within u32 words; e = p - (+-s)."""
    d, bucket = 1000, 128
    cfg = sign_cfg(d, bucket)
    g = rng(2).standard_normal(d).astype(np.float32)
    g[5] = -0.0
    g[6] = 0.0
    e = np.zeros(d, np.float32)
    msg = oracle.worker_step(cfg, 0, 1, g, e)
    off_s, off_p, total = oracle.layout(cfg)
    nb = -(-d // bucket)
    assert off_s == 0 and off_p == 256 * (-(-4 * nb // 256)) and total % 256 == 0
    scales = msg[off_s:off_s + 4 * nb].view(np.float32)
    words = msg[off_p:off_p + 4 * (-(-d // 32))].view(np.uint32)
    bits = np.unpackbits(words.view(np.uint8), bitorder="little")
    p = g  # lr = 1, e = 0
    np.testing.assert_array_equal(bits[:d].astype(bool), p < 0)
    assert not bits[d:].any()
    assert bits[5] == 0 and bits[6] == 0  # -0 and +0 both send +s
    # untouched padding stays zero
    assert not msg[4 * nb:off_p].any() and not msg[off_p + 4 * len(words):].any()
    for b in range(nb):
        blk = p[b * bucket:(b + 1) * bucket]
        assert scales[b] == oracle.sign_scale(blk, bucket)
        q = np.where(blk < 0, -scales[b], scales[b]).astype(np.float32)
        np.testing.assert_array_equal(e[b * bucket:(b + 1) * bucket], blk - q)


def test_sign_closed_form_and_delta_approximate():
    """||Q(x) - x||^2 = ||x||^2 - ||x||_1^2 / n per bucket (Definition 1 with delta >= 1/n)."""
    d, bucket = 4096 + 700, 512
    cfg = sign_cfg(d, bucket)
    x = (rng(3).standard_normal(d) * np.exp(rng(4).uniform(-4, 1, d))).astype(np.float32)
    e = np.zeros(d, np.float32)
    msg = oracle.worker_step(cfg, 0, 1, x, e)
    q = oracle.decode(cfg, msg).astype(np.float64)
    x64 = x.astype(np.float64)
    for start in range(0, d, bucket):
        xb, qb = x64[start:start + bucket], q[start:start + bucket]
        n = xb.size
        resid = np.sum((qb - xb) ** 2)
        closed = np.sum(xb ** 2) - np.sum(np.abs(xb)) ** 2 / n
        assert abs(resid - closed) <= 1e-5 * np.sum(xb ** 2)
        assert resid <= (1 - 1 / n) * np.sum(xb ** 2) * (1 + 1e-6)
    # the residual kept by the worker is exactly x - Q(x)
    np.testing.assert_array_equal(e, (x - q.astype(np.float32)))


@pytest.mark.parametrize("d", [3, 7, 10, 12])
def test_sign_brute_force_minimises_residual(d):
    """Among all sign patterns with their best scale, sign(x) with s = ||x||_1/d is optimal."""
    x = exact.frac_vec(rng(d).standard_normal(d).astype(np.float32))
    best = None
    for sigma in itertools.product((-1, 1), repeat=d):
        c = sum(s * v for s, v in zip(sigma, x)) / d
        r = sum((c * s - v) ** 2 for s, v in zip(sigma, x))
        best = r if best is None or r < best else best
    q = exact.q_sign(x, bucket=32)
    assert sum((a - b) ** 2 for a, b in zip(q, x)) == best
    # and the fp32 oracle's Q agrees with the exact one to rounding
    cfg = sign_cfg(d, 32)
    msg = oracle.worker_step(cfg, 0, 1, np.array([float(v) for v in x], np.float32),
                             np.zeros(d, np.float32))
    qo = oracle.decode(cfg, msg)
    for a, b in zip(qo, q):
        assert abs(Fraction(float(a)) - b) <= 4 * Fraction(U32) * abs(b)


# ---------------------------------------------------------------------------
# top-k
# ---------------------------------------------------------------------------

def topk_cfg(d, k, M=1, lr=1.0):
    return oracle.Config(d=d, M=M, compressor=oracle.TOPK, lr=lr, k=k)


@pytest.mark.parametrize("d,k", [(6, 1), (8, 3), (10, 5), (12, 4), (12, 12)])
def test_topk_brute_force_and_tie_rule(d, k):
    """The selection minimises ||Q(x)-x||^2 over all C(d,k) subsets and is the
    lexicographically smallest minimiser (ties to the lower index)."""
    r = rng(d * 31 + k)
    x = r.integers(-3, 4, size=d).astype(np.float32)  # small integers: many ties
    sel = oracle.topk_select(x, k)
    x64 = x.astype(np.float64)
    best, best_set = None, None
    for subset in itertools.combinations(range(d), k):
        resid = sum(x64[j] ** 2 for j in range(d) if j not in subset)
        if best is None or resid < best:
            best, best_set = resid, subset
    assert sel.sum() == k
    assert sum(x64[j] ** 2 for j in range(d) if not sel[j]) == best
    assert tuple(np.flatnonzero(sel)) == best_set


def test_topk_theorem1_and_message():
    d, k = 5000, 123
    cfg = topk_cfg(d, k)
    x = (rng(5).standard_normal(d) * np.exp(rng(6).uniform(-5, 2, d))).astype(np.float32)
    e = np.zeros(d, np.float32)
    msg = oracle.worker_step(cfg, 0, 1, x, e)
    rec = msg[:8 * k].view(np.uint32).reshape(k, 2)
    idx = rec[:, 0]
    vals = rec[:, 1].view(np.float32)
    assert np.all(np.diff(idx.astype(np.int64)) > 0)
    np.testing.assert_array_equal(vals, x[idx])
    # the k largest magnitudes
    thresh = np.sort(np.abs(x))[-k]
    assert np.all(np.abs(x[idx]) >= thresh)
    # Theorem 1: ||Q(x) - x||^2 <= (1 - k/d) ||x||^2
    q = oracle.decode(cfg, msg).astype(np.float64)
    assert np.sum((q - x) ** 2) <= (1 - k / d) * np.sum(x.astype(np.float64) ** 2)
    expect_e = x.copy()
    expect_e[idx] = 0.0
    np.testing.assert_array_equal(e, expect_e)
    assert not np.signbit(e[idx]).any()


def test_topk_degenerate_cases():
    d = 64
    # k = d: Q is the identity and the residual vanishes
    x = rng(7).standard_normal(d).astype(np.float32)
    e = np.zeros(d, np.float32)
    cfg = topk_cfg(d, d)
    msg = oracle.worker_step(cfg, 0, 1, x, e)
    np.testing.assert_array_equal(oracle.decode(cfg, msg), x)
    assert not e.any()
    # all-equal magnitudes: the first k indices win
    x = np.full(d, -2.0, np.float32)
    x[::2] = 2.0
    assert list(np.flatnonzero(oracle.topk_select(x, 5))) == [0, 1, 2, 3, 4]
    # zeros (both signs) tie with each other
    x = np.zeros(d, np.float32)
    x[10] = -0.0
    x[20] = 1e-30
    assert list(np.flatnonzero(oracle.topk_select(x, 3))) == [0, 1, 20]


# ---------------------------------------------------------------------------
# b-bit stochastic quantiser (proof of Theorem 2)
# ---------------------------------------------------------------------------

def squant_cfg(d, bits, bucket=512, M=1, lr=1.0, seed=99):
    return oracle.Config(d=d, M=M, compressor=oracle.SQUANT, lr=lr, bucket=bucket, bits=bits,
                         seed=seed)


@pytest.mark.parametrize("bits", [2, 4, 8])
def test_squant_moments_by_exact_enumeration(bits):
    """E[Q(v_i)] = v_i and E|Q(v_i)|^2 = |v_i| s (B_r + B_{r+1}) - B_r B_{r+1} s^2
    (proof of Theorem 2), enumerating both outcomes of every element of a
    bucket with their exact probabilities."""
    K = 2 ** (bits - 1) - 1
    n = 12
    v = exact.frac_vec(rng(bits).standard_normal(n).astype(np.float32))
    s = max(abs(x) for x in v)
    q_up = exact.q_squant(v, n, bits, [Fraction(0)] * n)   # u = 0 < f: every element rounds up
    q_dn = exact.q_squant(v, n, bits, [Fraction(1)] * n)   # u = 1 never rounds up
    for i, x in enumerate(v):
        t = abs(x) * K / s
        f = t - t.numerator // t.denominator
        r = t.numerator // t.denominator
        B_r, B_r1 = Fraction(r, K), Fraction(min(r + 1, K), K)
        p_up = f if f > 0 else Fraction(0)
        mean = p_up * q_up[i] + (1 - p_up) * q_dn[i]
        second = p_up * q_up[i] ** 2 + (1 - p_up) * q_dn[i] ** 2
        assert mean == x
        assert second == abs(x) * s * (B_r + B_r1) - B_r * B_r1 * s * s
        assert abs(q_dn[i]) == s * B_r and (f == 0 or abs(q_up[i]) == s * B_r1)


@pytest.mark.parametrize("bits", [2, 4, 8])
def test_squant_oracle_codes_match_exact_rule(bits):
    """With the oracle's own Philox draws, the fp32 codes follow the exact rounding rule."""
    d, bucket, seed = 3000, 512, 7
    cfg = squant_cfg(d, bits, bucket, seed=seed)
    x = (rng(bits + 10).standard_normal(d) * np.exp(rng(11).uniform(-3, 1, d))).astype(np.float32)
    e = np.zeros(d, np.float32)
    msg = oracle.worker_step(cfg, 5, 9, x, e)
    off_s, off_p, _ = oracle.layout(cfg)
    K = 2 ** (bits - 1) - 1
    nb = -(-d // bucket)
    scales = msg[off_s:off_s + 4 * nb].view(np.float32)
    words = msg[off_p:].view(np.uint32)
    codes = np.array([(int(words[(j * bits) >> 5]) >> ((j * bits) & 31)) & ((1 << bits) - 1)
                      for j in range(d)])
    assert codes.min() >= 0 and codes.max() <= 2 * K
    mismatches = 0
    for b in range(nb):
        blk = x[b * bucket:(b + 1) * bucket]
        assert scales[b] == np.max(np.abs(blk))
        s = Fraction(float(scales[b]))
        for off, xv in enumerate(blk):
            j = b * bucket + off
            u = Fraction(oracle.squant_uniform(seed, 5, 9, j))
            t = abs(Fraction(float(xv))) * K / s
            r = t.numerator // t.denominator
            level = min(r + (1 if u < t - r else 0), K)
            want = K - level if xv < 0 else K + level
            if codes[j] != want:
                mismatches += 1
                # only where fp32 rounding of |x| * (K/s) moved t across a boundary
                assert abs(codes[j] - want) == 1
    assert mismatches <= max(2, d // 500)
    # decode and residual
    q = oracle.decode(cfg, msg)
    np.testing.assert_array_equal(e, x - q)
    for j in range(0, d, 97):
        assert q[j] == oracle.squant_decode(int(codes[j]), float(scales[j // bucket]), K)


@pytest.mark.parametrize("bits", [4, 8])
def test_squant_unbiased_and_delta_over_philox_streams(bits):
    """Monte Carlo over 2048 steps: the mean of Q(v) is v (within 5 sigma) and
    E||Q(v) - v||^2 <= (1 - delta) ||v||^2 with delta > 0 for b = 4, 8."""
    d, bucket = 64, 64
    cfg = squant_cfg(d, bits, bucket, seed=12345)
    v = (rng(20 + bits).standard_normal(d)).astype(np.float32)
    T = 2048
    qs = np.empty((T, d), np.float64)
    for t in range(T):
        msg = oracle.worker_step(cfg, 0, t + 1, v, np.zeros(d, np.float32))
        qs[t] = oracle.decode(cfg, msg)
    K = 2 ** (bits - 1) - 1
    s = float(np.max(np.abs(v)))
    mean = qs.mean(0)
    sd = s / K / 2  # per-element std of a two-point draw is at most half a level
    assert np.all(np.abs(mean - v) <= 5 * sd / math.sqrt(T) + 1e-6)
    # second moment against the closed form of Theorem 2's proof
    a = np.abs(v.astype(np.float64))
    r = np.floor(a * K / s)
    lo, hi = r / K, np.minimum(r + 1, K) / K
    closed = a * s * (lo + hi) - lo * hi * s * s
    emp = (qs ** 2).mean(0)
    assert np.all(np.abs(emp - closed) <= 6 * s * s / math.sqrt(T) + 1e-6)
    ratio = np.sum((qs - v) ** 2, 1).mean() / np.sum(v.astype(np.float64) ** 2)
    assert ratio < 1.0


def test_squant_two_bit_is_not_delta_approximate_on_gaussians():
    """The proof of Theorem 2 needs 3 C_r > C_{r+1}, which fails at r = 0; with
    b = 2 (levels 0, s) the expected residual exceeds ||v||^2 on Gaussian
    buckets.  The measured ratio is recorded rather than asserted below 1."""
    d = 512
    cfg = squant_cfg(d, 2, 512, seed=3)
    v = rng(30).standard_normal(d).astype(np.float32)
    T = 256
    tot = 0.0
    for t in range(T):
        msg = oracle.worker_step(cfg, 0, t + 1, v, np.zeros(d, np.float32))
        q = oracle.decode(cfg, msg).astype(np.float64)
        tot += np.sum((q - v) ** 2)
    ratio = tot / T / np.sum(v.astype(np.float64) ** 2)
    s = np.max(np.abs(v))
    expected = (s * np.sum(np.abs(v)) - np.sum(v.astype(np.float64) ** 2)) / np.sum(v.astype(np.float64) ** 2)
    assert abs(ratio - expected) < 0.05 * expected
    assert ratio > 1.0


def test_squant_zero_bucket_and_extremes():
    d, bits, bucket = 1024, 4, 512
    cfg = squant_cfg(d, bits, bucket)
    x = rng(40).standard_normal(d).astype(np.float32)
    x[:512] = 0.0
    x[3] = -0.0
    e = np.zeros(d, np.float32)
    msg = oracle.worker_step(cfg, 0, 1, x, e)
    q = oracle.decode(cfg, msg)
    K = 7
    off_s, off_p, _ = oracle.layout(cfg)
    assert msg[0:4].view(np.float32)[0] == 0.0
    words = msg[off_p:].view(np.uint32)
    assert all(((int(words[(j * bits) >> 5]) >> ((j * bits) & 31)) & 15) == K for j in range(512))
    assert not q[:512].any() and np.array_equal(e[:512], x[:512])
    # the bucket maximum always decodes to +-s exactly
    jmax = 512 + int(np.argmax(np.abs(x[512:])))
    assert abs(q[jmax]) == np.max(np.abs(x[512:])) and np.sign(q[jmax]) == np.sign(x[jmax])


# ---------------------------------------------------------------------------
# Algorithm 2 as a whole
# ---------------------------------------------------------------------------

def test_error_feedback_telescopes():
    """Appendix B, error-corrected sequence: sum_t Q(p_t) + e_T = sum_t eta g_t
    for every worker (within fp32 rounding of the running sums)."""
    d, M, T = 2048, 3, 12
    for comp, extra in [(oracle.SIGN, {"bucket": 256}), (oracle.TOPK, {"k": 100}),
                        (oracle.SQUANT, {"bucket": 256, "bits": 4})]:
        cfg = oracle.Config(d=d, M=M, compressor=comp, lr=0.01, **extra)
        st = oracle.State(cfg)
        sent = np.zeros((M, d), np.float64)
        fed = np.zeros((M, d), np.float64)
        bound = np.zeros((M, d), np.float64)
        w = np.zeros(d, np.float32)
        for t in range(T):
            g = (rng(100 + t).standard_normal((M, d))).astype(np.float32)
            msgs = st.step(g, w)
            for i in range(M):
                q = oracle.decode(cfg, msgs[i]).astype(np.float64)
                sent[i] += q
                fed[i] += (np.float32(cfg.lr) * g[i]).astype(np.float64)
                bound[i] += 4 * U32 * (np.abs(q) + np.abs(fed[i]) + np.abs(st.e[i]))
        lhs = sent + st.e.astype(np.float64)
        assert np.all(np.abs(lhs - fed) <= bound + 1e-12), comp


def test_error_feedback_telescopes_exactly_in_rationals():
    """Same identity with no rounding at all (exact replay)."""
    d, M, T = 9, 2, 6
    r = rng(50)
    grads = {(m, t): exact.frac_vec(r.standard_normal(d).astype(np.float32))
             for m in range(M) for t in range(1, T + 1)}
    for compress in (lambda p, m, t: exact.q_sign(p, 4), lambda p, m, t: exact.q_topk(p, 3)):
        alg = exact.ExactDQGAN([Fraction(0)] * d, M, Fraction(1, 8), compress)
        for _ in range(T):
            alg.step(lambda m, t, w: grads[(m, t)])
        for m in range(M):
            sent = [sum((rec["p_hat"][m][j] for rec in alg.history), Fraction(0)) for j in range(d)]
            fed = [sum((Fraction(1, 8) * grads[(m, t)][j] for t in range(1, T + 1)), Fraction(0))
                   for j in range(d)]
            assert [a + b for a, b in zip(sent, alg.e[m])] == fed


def test_lemma1_per_step_contraction():
    """||e_t||^2 <= (1 - delta) ||p_t||^2 at every step and worker (proof of Lemma 1),
    delta = 1/n for the scaled sign and k/d for top-k."""
    d, M, T = 4096, 2, 8
    for comp, extra, delta in [(oracle.SIGN, {"bucket": 512}, 1 / 512),
                               (oracle.TOPK, {"k": 64}, 64 / 4096)]:
        cfg = oracle.Config(d=d, M=M, compressor=comp, lr=0.05, **extra)
        st = oracle.State(cfg)
        w = np.zeros(d, np.float32)
        for t in range(T):
            g = (rng(200 + t).standard_normal((M, d)) * 3).astype(np.float32)
            p = [(np.float32(cfg.lr) * g[i] + st.e[i]).astype(np.float32) for i in range(M)]
            st.step(g, w)
            for i in range(M):
                pe = np.sum(p[i].astype(np.float64) ** 2)
                ee = np.sum(st.e[i].astype(np.float64) ** 2)
                assert ee <= (1 - delta) * pe * (1 + 1e-6)


def test_identity_reduces_to_uncompressed_distributed_omd():
    """With Q = identity the residual stays zero and w_t = w_{t-1} - (1/M) sum_m eta g_m."""
    d, M, T = 777, 4, 5
    cfg = oracle.Config(d=d, M=M, compressor=oracle.IDENTITY, lr=0.125)
    st = oracle.State(cfg)
    w = rng(60).standard_normal(d).astype(np.float32)
    w_exact = exact.frac_vec(w)
    for t in range(T):
        g = rng(61 + t).standard_normal((M, d)).astype(np.float32)
        st.step(g, w)
        assert not st.e.any()
        upd = [sum((Fraction(float(np.float32(cfg.lr) * g[m, j])) for m in range(M)), Fraction(0)) / M
               for j in range(d)]
        w_exact = [a - b for a, b in zip(w_exact, upd)]
        err = max(abs(Fraction(float(a)) - b) for a, b in zip(w, w_exact))
        scale = max(abs(b) for b in w_exact)
        assert err <= (t + 1) * 8 * Fraction(U32) * (scale + 1)


# ---------------------------------------------------------------------------
# The server's sum over workers.  Algorithm 2 averages the M decoded messages;
# the paper leaves the order of the sum open, and the reading taken fixes it
# to pairwise summation over the M values padded with +0 to a power of two.
# Two facts of the mathematics pin that order: (1) pairwise summation's
# forward error is at most ceil(log2 M) u sum|x| (Higham, Accuracy and
# Stability of Numerical Algorithms, section 4.2), a bound that recursive
# (worker-order) summation breaks on adversarial inputs; (2) where every
# pairwise partial sum is exact, the average is the exact average.
# ---------------------------------------------------------------------------
U_HALF = 2.0 ** -24  # unit roundoff of binary32


@pytest.mark.parametrize("M", [2, 3, 5, 8, 13, 16, 33, 64, 100])
def test_server_sum_is_within_the_pairwise_error_bound(M):
    r = rng(90 + M)
    cases = [r.standard_normal(M), np.abs(r.standard_normal(M)) * 2.0 ** r.integers(-20, 20, M),
             np.concatenate([[1.0], np.full(M - 1, U_HALF)])]
    levels = int(np.ceil(np.log2(M)))
    for x in cases:
        x = np.asarray(x, np.float32)
        exact_sum = sum((Fraction(float(v)) for v in x), Fraction(0))
        got = Fraction(oracle.pairwise_sum(x))
        bound = Fraction(levels) * Fraction(U_HALF) * sum(abs(Fraction(float(v))) for v in x)
        assert abs(got - exact_sum) <= bound * (1 + Fraction(1, 10 ** 6)), (M, float(got), float(exact_sum))


def test_worker_order_summation_would_break_the_bound():
    """The adversarial input of the test above separates the orders: adding
    63 halves of an ulp to 1 one at a time loses every one of them."""
    x = np.concatenate([[1.0], np.full(63, U_HALF)]).astype(np.float32)
    seq = np.float32(0.0)
    for v in x:
        seq = np.float32(seq + v)
    exact_sum = Fraction(1) + 63 * Fraction(U_HALF)
    bound = 6 * Fraction(U_HALF) * exact_sum
    assert abs(Fraction(float(seq)) - exact_sum) > bound
    assert abs(Fraction(oracle.pairwise_sum(x)) - exact_sum) <= bound


@pytest.mark.parametrize("vals", [(1.0, 0.0, U_HALF, U_HALF), (1.0, 0.0, 0.0, 0.0) + (U_HALF,) * 4,
                                  (0.0, 0.0, 1.0, 0.0, 2 * U_HALF, 0.0, 2 * U_HALF, 0.0)])
def test_server_average_is_exact_when_pairwise_partial_sums_are(vals):
    """Identity messages carrying these values per element: the exact
    average sum/M is representable and every pairwise partial sum is exact,
    so the server must subtract exactly sum/M (a worker-order sum would drop
    the small terms against the 1)."""
    M, d = len(vals), 8
    cfg = oracle.Config(d=d, M=M, compressor=oracle.IDENTITY)
    msgs = np.zeros((M, oracle.message_bytes(cfg)), np.uint8)
    for m, v in enumerate(vals):
        msgs[m, :4 * d] = np.full(d, v, np.float32).view(np.uint8)
    w = np.zeros(d, np.float32)
    oracle.server_step(cfg, msgs, w)
    want = -(sum((Fraction(float(np.float32(v))) for v in vals), Fraction(0)) / M)
    assert all(Fraction(float(x)) == want for x in w), (w[0], float(want))


def test_pairwise_sum_pads_with_positive_zero():
    """A power-of-two count is not padded (one -0 stays -0); any other count
    adds +0 leaves, which turn a -0 partial sum into +0."""
    assert math.copysign(1.0, oracle.pairwise_sum([-0.0])) < 0
    assert math.copysign(1.0, oracle.pairwise_sum([-0.0, -0.0])) < 0
    three = oracle.pairwise_sum([-0.0, -0.0, -0.0])
    assert three == 0.0 and math.copysign(1.0, three) > 0
    # the padding is exactly zero: the smallest subnormal survives it
    tiny = 2.0 ** -149
    assert oracle.pairwise_sum([tiny, 0.0, 0.0]) == tiny
    assert oracle.pairwise_sum([-tiny] * 5) == -5 * tiny


def bilinear_F(w):
    """F(x, y) = (y, -x): the operator of the bilinear game min_x max_y x.y."""
    half = len(w) // 2
    return list(w[half:]) + [-v for v in w[:half]]


def test_single_worker_identity_obeys_one_line_omd():
    """M = 1, Q = identity: w_{t+1/2} = w_{t-1/2} - 2 eta F(w_{t-1/2}) + eta F(w_{t-3/2})."""
    d = 6
    lr = Fraction(1, 10)
    w0 = exact.frac_vec([1, -2, 0.5, 3, -1, 2])
    alg = exact.ExactDQGAN(w0, 1, lr, lambda p, m, t: exact.q_identity(p))
    F = lambda m, t, w: bilinear_F(w)
    halves, grads = [], []
    for _ in range(6):
        rec = alg.step(F)
        halves.append(rec["w_half"][0])
        grads.append(rec["F"][0])
    for t in range(1, 5):
        F_prev = grads[t - 1]
        want = [a - 2 * lr * b + lr * c for a, b, c in zip(halves[t], grads[t], F_prev)]
        assert halves[t + 1] == want
    # t = 1 convention: F(w_{-1/2}) := 0, so w_{1/2} = w_0
    assert halves[0] == w0


def test_fp32_oracle_equals_exact_replay_on_dyadic_inputs():
    """Where no operation rounds (dyadic inputs, power-of-two bucket and M),
    the fp32 oracle and the exact replay agree bit for bit over 5 steps."""
    d, M, T = 16, 2, 5
    r = rng(70)
    grads = {(m, t): [Fraction(int(v), 16) for v in r.integers(-64, 65, size=d)]
             for m in range(M) for t in range(1, T + 1)}
    cases = [
        (oracle.SIGN, {"bucket": 4}, lambda p, m, t: exact.q_sign(p, 4)),
        (oracle.TOPK, {"k": 5}, lambda p, m, t: exact.q_topk(p, 5)),
        (oracle.IDENTITY, {}, lambda p, m, t: exact.q_identity(p)),
    ]
    for comp, extra, qfun in cases:
        cfg = oracle.Config(d=d, M=M, compressor=comp, lr=1.0, keep_lookahead=True, **extra)
        st = oracle.State(cfg)
        w = np.array([float(x) for x in exact.frac_vec(np.arange(d) / 8 - 1)], np.float32)
        alg = exact.ExactDQGAN(exact.frac_vec(w), M, Fraction(1), qfun)
        for t in range(1, T + 1):
            g = np.array([[float(v) for v in grads[(m, t)]] for m in range(M)], np.float32)
            w_half = [oracle.lookahead(w, st.h[m]) for m in range(M)]
            rec = alg.step(lambda m, tt, wh: grads[(m, tt)])
            for m in range(M):
                assert [Fraction(float(v)) for v in w_half[m]] == rec["w_half"][m]
            st.step(g, w)
            assert [Fraction(float(v)) for v in w] == rec["w"], (comp, t)
            for m in range(M):
                assert [Fraction(float(v)) for v in st.e[m]] == rec["e"][m]


def test_squant_fp32_equals_exact_on_dyadic_single_step():
    """b = 2 (K = 1) with a power-of-two bucket maximum: one step is exact."""
    d, bucket = 32, 8
    cfg = squant_cfg(d, 2, bucket, seed=77)
    r = rng(80)
    x = r.integers(-15, 16, size=d).astype(np.float32) / 16
    for b in range(0, d, bucket):
        x[b + 3] = -1.0  # bucket max |x| = 1
    e = np.zeros(d, np.float32)
    msg = oracle.worker_step(cfg, 2, 4, x, e)
    us = [Fraction(oracle.squant_uniform(77, 2, 4, j)) for j in range(d)]
    q_exact = exact.q_squant(exact.frac_vec(x), bucket, 2, us)
    q = oracle.decode(cfg, msg)
    assert [Fraction(float(v)) for v in q] == q_exact
    assert [Fraction(float(v)) for v in e] == [a - b for a, b in zip(exact.frac_vec(x), q_exact)]


def test_bilinear_game_lookahead_converges_where_plain_step_spirals():
    """Section 2.2: on min_x max_y x.y plain simultaneous steps drift away while
    the optimistic (lookahead) step of Algorithm 2 contracts, also with the
    compressed, error-compensated messages."""
    d, M, T = 64, 2, 400
    lr = 0.1
    w_init = rng(90).standard_normal(d).astype(np.float32)

    def run(lookahead: bool, comp: int):
        cfg = oracle.Config(d=d, M=M, compressor=comp, lr=lr, bucket=32, keep_lookahead=True)
        st = oracle.State(cfg)
        w = w_init.copy()
        for _ in range(T):
            g = np.empty((M, d), np.float32)
            for m in range(M):
                wh = oracle.lookahead(w, st.h[m]) if lookahead else w
                g[m] = np.concatenate([wh[d // 2:], -wh[:d // 2]])
            st.step(g, w)
        return float(np.linalg.norm(w))

    n0 = float(np.linalg.norm(w_init))
    # plain steps grow the norm by sqrt(1 + lr^2) per step: 7.3x after 400 steps
    assert run(False, oracle.IDENTITY) > 5 * n0
    assert run(False, oracle.SIGN) > 5 * n0
    assert run(True, oracle.IDENTITY) < 0.25 * n0
    assert run(True, oracle.SIGN) < 0.25 * n0


# ---------------------------------------------------------------------------
# QSGD: the b-bit stochastic quantiser with the l2 scale (Section 2.4, Eq. (qsgd))
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("bucket", [32, 512, 4096])
@pytest.mark.parametrize("count_frac", [1.0, 0.41])
def test_qsgd_scale_is_the_l2_norm(bucket, count_frac):
    count = max(1, int(bucket * count_frac))
    x = (rng(bucket * 7 + count).standard_normal(count) * np.exp(rng(count + 1).uniform(-6, 2, count)))
    x = x.astype(np.float32)
    got = Fraction(oracle.qsgd_sumsq(x, bucket))
    want = exact.sq_norm(exact.frac_vec(x))
    # every square rounds once and every addition once: (n + 1) u relative
    assert abs(got - want) <= Fraction(count + 1) * Fraction(U32) * want * Fraction(11, 10)
    s = oracle.qsgd_scale(x, bucket)
    assert s == np.float32(np.sqrt(np.float32(oracle.qsgd_sumsq(x, bucket))))
    assert abs(s - math.sqrt(float(want))) <= 4 * U32 * s
    for j in [0, count // 3, count - 1]:
        y = x.copy()
        y[j] = np.float32(1e5)
        assert oracle.qsgd_sumsq(y, bucket) >= 1e10


@pytest.mark.parametrize("bits", [2, 4, 8])
def test_qsgd_moments_by_exact_enumeration(bits):
    """With the l2 scale (>= every |v_i|) the quantiser is unbiased and has the
    second moment of the proof of Theorem 2, element by element."""
    K = 2 ** (bits - 1) - 1
    n = 10
    v32 = rng(40 + bits).standard_normal(n).astype(np.float32)
    s = Fraction(oracle.qsgd_scale(v32, 16))
    v = exact.frac_vec(v32)
    assert all(abs(x) <= s for x in v)
    q_up = exact.q_squant(v, n, bits, [Fraction(0)] * n, scales=[s])
    q_dn = exact.q_squant(v, n, bits, [Fraction(1)] * n, scales=[s])
    for i, x in enumerate(v):
        t = abs(x) * K / s
        r = t.numerator // t.denominator
        f = t - r
        B_r, B_r1 = Fraction(r, K), Fraction(min(r + 1, K), K)
        mean = f * q_up[i] + (1 - f) * q_dn[i]
        second = f * q_up[i] ** 2 + (1 - f) * q_dn[i] ** 2
        assert mean == x
        assert second == abs(x) * s * (B_r + B_r1) - B_r * B_r1 * s * s


@pytest.mark.parametrize("bits", [2, 4, 8])
def test_qsgd_oracle_codes_match_exact_rule(bits):
    d, bucket, seed = 2000, 256, 9
    cfg = oracle.Config(d=d, M=1, compressor=oracle.QSGD, lr=1.0, bucket=bucket, bits=bits, seed=seed)
    x = (rng(bits + 50).standard_normal(d) * np.exp(rng(51).uniform(-3, 1, d))).astype(np.float32)
    e = np.zeros(d, np.float32)
    msg = oracle.worker_step(cfg, 2, 6, x, e)
    off_s, off_p, _ = oracle.layout(cfg)
    K = 2 ** (bits - 1) - 1
    nb = -(-d // bucket)
    scales = msg[off_s:off_s + 4 * nb].view(np.float32)
    words = msg[off_p:].view(np.uint32)
    mismatches = 0
    for b in range(nb):
        blk = x[b * bucket:(b + 1) * bucket]
        assert scales[b] == np.float32(oracle.qsgd_scale(blk, bucket))
        s = Fraction(float(scales[b]))
        for off, xv in enumerate(blk):
            j = b * bucket + off
            code = (int(words[(j * bits) >> 5]) >> ((j * bits) & 31)) & ((1 << bits) - 1)
            u = Fraction(oracle.squant_uniform(seed, 2, 6, j))
            t = abs(Fraction(float(xv))) * K / s
            r = t.numerator // t.denominator
            level = min(r + (1 if u < t - r else 0), K)
            want = K - level if xv < 0 else K + level
            if code != want:
                mismatches += 1
                assert abs(code - want) == 1
    assert mismatches <= max(2, d // 500)
    np.testing.assert_array_equal(e, x - oracle.decode(cfg, msg))


@pytest.mark.parametrize("bits", [4, 8])
def test_qsgd_unbiased_and_variance_bound_over_philox_streams(bits):
    """Monte Carlo over 2048 steps: mean of Q(v) is v, and the expected residual
    respects QSGD's variance bound min(n/K^2, sqrt(n)/K) ||v||^2 (Alistarh et
    al., the compressor Eq. (qsgd) cites) and is below ||v||^2 (delta > 0)."""
    n = 64
    cfg = oracle.Config(d=n, M=1, compressor=oracle.QSGD, lr=1.0, bucket=n, bits=bits, seed=321)
    v = rng(60 + bits).standard_normal(n).astype(np.float32)
    T = 2048
    qs = np.empty((T, n), np.float64)
    for t in range(T):
        qs[t] = oracle.decode(cfg, oracle.worker_step(cfg, 0, t + 1, v, np.zeros(n, np.float32)))
    K = 2 ** (bits - 1) - 1
    s = float(np.linalg.norm(v.astype(np.float64)))
    assert np.all(np.abs(qs.mean(0) - v) <= 5 * (s / K / 2) / math.sqrt(T) + 1e-6)
    resid = np.sum((qs - v) ** 2, 1).mean()
    vv = np.sum(v.astype(np.float64) ** 2)
    assert resid <= min(n / K ** 2, math.sqrt(n) / K) * vv * 1.1
    assert resid < vv


# --- per-layer-segment bucketing (buckets restart at every layer boundary) ---

def _py_bucket_starts(segments, bucket):
    starts = []
    for a, b in zip(segments[:-1], segments[1:]):
        starts.extend(range(a, b, bucket))
    return starts + [segments[-1]]


def _random_segments(rng, d, n):
    cuts = np.sort(rng.choice(np.arange(1, d // 32), size=n - 1, replace=False)) * 32
    return tuple([0, *cuts.tolist(), d])


SEG_CASES = [(5_000, 512, (0, 32, 64, 4_000, 5_000)), (4_131, 256, (0, 4_131)),
             (10_007, 1024, None), (3_000, 32, (0, 96, 2_048, 2_080, 3_000))]


@pytest.mark.parametrize("d,bucket,segs", SEG_CASES)
def test_segment_bucket_boundaries(d, bucket, segs):
    segs = segs if segs is not None else _random_segments(np.random.default_rng(d), d, 7)
    cfg = oracle.Config(d=d, M=1, compressor=oracle.SIGN, bucket=bucket, segments=segs)
    got = oracle.bucket_starts(cfg)
    assert got.tolist() == _py_bucket_starts(list(segs), bucket)
    _, off_p, total = oracle.layout(cfg)
    nb = len(got) - 1
    assert off_p == -(-4 * nb // 256) * 256
    assert total == -(-(off_p + 4 * (-(-d // 32))) // 256) * 256


@pytest.mark.parametrize("d,bucket,segs", SEG_CASES)
def test_segmented_sign_is_flat_sign_per_segment(d, bucket, segs):
    """The sign compressor is deterministic and bucket-local: with segments,
    each segment's scales and bits are those of the flat compressor run on
    that segment alone."""
    rng = np.random.default_rng(11)
    segs = segs if segs is not None else _random_segments(np.random.default_rng(d), d, 7)
    g = (rng.standard_normal(d) * np.exp(rng.uniform(-3, 2, d))).astype(np.float32)
    cfg = oracle.Config(d=d, M=1, compressor=oracle.SIGN, bucket=bucket, lr=0.5, segments=segs)
    e = np.zeros(d, np.float32)
    msg = oracle.worker_step(cfg, 0, 1, g, e)
    off_s, off_p, _ = oracle.layout(cfg)
    scales = msg[off_s:].view(np.float32)
    words = msg[off_p:].view(np.uint32)
    b = 0
    for a, z in zip(segs[:-1], segs[1:]):
        sub = oracle.Config(d=z - a, M=1, compressor=oracle.SIGN, bucket=bucket, lr=0.5)
        e_sub = np.zeros(z - a, np.float32)
        m_sub = oracle.worker_step(sub, 0, 1, g[a:z].copy(), e_sub)
        s_off, p_off, _ = oracle.layout(sub)
        nb_sub = -(-(z - a) // bucket)
        assert np.array_equal(scales[b:b + nb_sub].view(np.uint32),
                              m_sub[s_off:s_off + 4 * nb_sub].view(np.uint32))
        bits_seg = np.unpackbits(words.view(np.uint8), bitorder="little")[a:z]
        bits_sub = np.unpackbits(m_sub[p_off:].view(np.uint8), bitorder="little")[:z - a]
        assert np.array_equal(bits_seg, bits_sub)
        assert_array_bits(e[a:z], e_sub)
        b += nb_sub


def assert_array_bits(x, y):
    assert np.array_equal(np.asarray(x, np.float32).view(np.uint32), np.asarray(y, np.float32).view(np.uint32))


@pytest.mark.parametrize("comp", [oracle.SQUANT, oracle.QSGD])
@pytest.mark.parametrize("d,bucket,segs", SEG_CASES)
def test_segmented_quantiser_scales_and_levels(comp, d, bucket, segs):
    """Each bucket's scale is the max (or the l2 norm) over exactly its own
    elements, and every decoded value is a level of that bucket's scale
    bracketing |p_j| (Section 2.4, proof of Theorem 2)."""
    rng = np.random.default_rng(5)
    segs = segs if segs is not None else _random_segments(np.random.default_rng(d), d, 7)
    bits = 4
    K = 2 ** (bits - 1) - 1
    g = (rng.standard_normal(d) * np.exp(rng.uniform(-3, 2, d))).astype(np.float32)
    cfg = oracle.Config(d=d, M=1, compressor=comp, bucket=bucket, bits=bits, lr=1.0, seed=9, segments=segs)
    e = np.zeros(d, np.float32)
    msg = oracle.worker_step(cfg, 0, 3, g, e)
    p = g.astype(np.float64)
    q = oracle.decode(cfg, msg).astype(np.float64)
    starts = _py_bucket_starts(list(segs), bucket)
    scales = msg[oracle.layout(cfg)[0]:].view(np.float32)
    for b in range(len(starts) - 1):
        blk = p[starts[b]:starts[b + 1]]
        want = np.max(np.abs(blk)) if comp == oracle.SQUANT else np.sqrt(np.sum(blk * blk))
        assert abs(scales[b] - want) <= 1e-6 * want + 1e-30, (b, scales[b], want)
        s = float(scales[b])
        lv = np.abs(q[starts[b]:starts[b + 1]]) / s * K
        t = np.abs(blk) / s * K
        assert np.all(np.abs(lv - np.round(lv)) < 1e-4)
        assert np.all(np.round(lv) >= np.floor(t * (1 - 1e-6)) - 1e-9)
        assert np.all(np.round(lv) <= np.ceil(t * (1 + 1e-6)) + 1e-9)


@pytest.mark.parametrize("comp", [oracle.SIGN, oracle.SQUANT, oracle.QSGD])
def test_one_segment_is_the_flat_layout(comp):
    rng = np.random.default_rng(2)
    d = 9_001
    g = rng.standard_normal((2, d)).astype(np.float32)
    out = []
    for segs in (None, (0, d)):
        cfg = oracle.Config(d=d, M=2, compressor=comp, bucket=512, bits=8, lr=0.1, seed=4, segments=segs)
        st = oracle.State(cfg)
        w = np.zeros(d, np.float32)
        out.append((st.step(g, w), w))
    assert np.array_equal(out[0][0], out[1][0])
    assert np.array_equal(out[0][1], out[1][1])


# ---------------------------------------------------------------------------
# Optimistic Adam server update (the CPOAdam family of Section 4; the rule of
# Daskalakis et al., ICLR 2018, fed the averaged update q_hat).
# ---------------------------------------------------------------------------

def dyadic(r, shape, bits=8, scale=1.0):
    """Random values with at most `bits` significant bits (products and squares stay exact in fp32)."""
    ints = r.integers(-(2 ** bits) + 1, 2 ** bits, size=shape)
    ints[ints == 0] = 1
    return (ints.astype(np.float64) * scale / 2 ** bits).astype(np.float32)


def test_oadam_reduces_to_the_one_line_omd_recurrence():
    """b1 = 0, identity preconditioner, alpha = 1, one worker, identity Q, the
    gradient taken at the current iterate: Algorithm 2's server with this
    update obeys w_{t+1} = w_t - 2 eta F(w_t) + eta F(w_{t-1}) (Section 2.2)
    exactly (dyadic data: no operation rounds)."""
    d, T = 8, 6
    lr = 0.125
    cfg = oracle.Config(d=d, M=1, compressor=oracle.IDENTITY, lr=lr)
    st = oracle.State(cfg)
    opt = oracle.OAdamState(d, oracle.OAdam(alpha=1.0, beta1=0.0, beta2=0.0, eps=0.0, adaptive=False,
                                            bias_correction=False))
    w = dyadic(rng(100), d, bits=6)
    w_exact = exact.frac_vec(w)
    F_prev = [Fraction(0)] * d
    for t in range(1, T + 1):
        F = bilinear_F(w_exact)
        g = np.array([float(x) for x in F], np.float32)
        msgs = st.compress_all(g[None, :])
        q_hat = oracle.server_average(cfg, msgs)
        opt.update(t, q_hat, w)
        st.t += 1
        w_exact = [x - 2 * Fraction(lr) * f + Fraction(lr) * fp for x, f, fp in zip(w_exact, F, F_prev)]
        F_prev = F
        assert [Fraction(float(x)) for x in w] == w_exact, t


def test_oadam_first_step_is_a_signed_step():
    """t = 1 with bias correction and eps = 0: m_hat = q, v_hat = q^2, so
    u = sign(q) and w_1 = w_0 - 2 alpha sign(q) exactly (dyadic b1, b2)."""
    d = 500
    r = rng(101)
    q = dyadic(r, d, bits=10, scale=2.0 ** -7)
    w0 = dyadic(r, d, bits=12)
    w = w0.copy()
    st = oracle.OAdamState(d, oracle.OAdam(alpha=0.0625, beta1=0.5, beta2=0.75, eps=0.0))
    st.update(1, q, w)
    assert np.array_equal(st.u, np.sign(q).astype(np.float32))
    assert np.array_equal(w, (w0 - np.float32(0.125) * np.sign(q)).astype(np.float32))


def test_oadam_matches_the_exact_replay():
    """b2 = 0 makes sqrt(v_hat) = |q| rational, so the rule can be replayed in
    exact arithmetic; the fp32 oracle stays within a few roundings of it over
    8 steps (adaptive and identity preconditioner, with and without bias
    correction)."""
    d, T = 16, 8
    for adaptive in (True, False):
        for bc in (True, False):
            r = rng(102)
            opt = oracle.OAdam(alpha=0.0625, beta1=0.75, beta2=0.0, eps=2.0 ** -6, adaptive=adaptive,
                               bias_correction=bc)
            st = oracle.OAdamState(d, opt)
            ex = exact.ExactOAdam(d, opt.alpha, opt.beta1, opt.beta2, opt.eps, adaptive, bc)
            w = dyadic(r, d, bits=10)
            w_ex = exact.frac_vec(w)
            for t in range(1, T + 1):
                q = dyadic(r, d, bits=6, scale=2.0 ** -3)
                st.update(t, q, w)
                w_ex = ex.update(t, exact.frac_vec(q), w_ex)
                scale = max(abs(x) for x in w_ex) + 1
                err = max(abs(Fraction(float(a)) - b) for a, b in zip(w, w_ex))
                assert err <= 64 * t * Fraction(U32) * scale, (adaptive, bc, t, float(err))


def test_oadam_is_invariant_to_power_of_two_gradient_scaling():
    """With eps = 0 the update u depends on q only through q / sqrt(E q^2):
    scaling every q by 2^k scales m by 2^k, v by 4^k and leaves u and w bit
    for bit unchanged (no operation rounds differently)."""
    d, T = 1000, 6
    qs = [(rng(103 + t).standard_normal(d) * 1e-3).astype(np.float32) for t in range(T)]
    w0 = rng(110).standard_normal(d).astype(np.float32)
    runs = []
    for k in (0, 7, -9):
        st = oracle.OAdamState(d, oracle.OAdam(alpha=1e-3, beta1=0.5, beta2=0.999, eps=0.0))
        w = w0.copy()
        for t, q in enumerate(qs, 1):
            st.update(t, (q * np.float32(2.0 ** k)).astype(np.float32), w)
        runs.append((w, st.u.copy()))
    for w, u in runs[1:]:
        assert np.array_equal(w.view(np.uint32), runs[0][0].view(np.uint32))
        assert np.array_equal(u.view(np.uint32), runs[0][1].view(np.uint32))


def test_oadam_is_odd_in_the_gradients():
    """Negating every q and w_0 negates m, u and w exactly and leaves v."""
    d, T = 777, 5
    qs = [(rng(120 + t).standard_normal(d)).astype(np.float32) for t in range(T)]
    w0 = rng(130).standard_normal(d).astype(np.float32)
    opt = oracle.OAdam(alpha=1e-2, beta1=0.9, beta2=0.99, eps=1e-6)
    a, b = oracle.OAdamState(d, opt), oracle.OAdamState(d, opt)
    wa, wb = w0.copy(), (-w0).astype(np.float32)
    for t, q in enumerate(qs, 1):
        a.update(t, q, wa)
        b.update(t, (-q).astype(np.float32), wb)
    assert np.array_equal(wb, -wa) and np.array_equal(b.u, -a.u) and np.array_equal(b.m, -a.m)
    assert np.array_equal(b.v, a.v)


@pytest.mark.parametrize("beta1,beta2", [(0.5, 0.999), (0.9, 0.999), (0.0, 0.9), (0.9, 0.99)])
def test_oadam_step_is_bounded(beta1, beta2):
    """Cauchy-Schwarz on m_t = (1-b1) sum b1^(t-s) q_s against
    v_t = (1-b2) sum b2^(t-s) q_s^2 bounds every update (eps = 0):
    |u_t| <= (1-b1) sqrt(S_t) sqrt(1-b2^t) / ((1-b1^t) sqrt(1-b2)),
    S_t = sum_{k<t} (b1^2/b2)^k -- for any gradients, heavy-tailed included."""
    d, T = 4000, 12
    r = rng(140)
    st = oracle.OAdamState(d, oracle.OAdam(alpha=1e-3, beta1=beta1, beta2=beta2, eps=0.0))
    w = np.zeros(d, np.float32)
    for t in range(1, T + 1):
        q = (r.standard_t(2, d) * 10.0 ** r.uniform(-4, 1, d)).astype(np.float32)
        st.update(t, q, w)
        S = sum((beta1 ** 2 / beta2) ** k for k in range(t))
        bound = (1 - beta1) * math.sqrt(S) * math.sqrt(1 - beta2 ** t) / ((1 - beta1 ** t) * math.sqrt(1 - beta2))
        assert np.max(np.abs(st.u)) <= bound * (1 + 1e-5), (t, float(np.max(np.abs(st.u))), bound)


def test_oadam_bias_correction_power_is_a_running_product():
    """b^t is the product of t factors: b^0 = 1, b^1 = b, and b^(t+1) = fl(b^t * b)."""
    for b in (0.9, 0.999, 0.5):
        assert oracle.pow_steps(b, 0) == 1.0 and oracle.pow_steps(b, 1) == np.float32(b)
        for t in (2, 7, 100):
            assert oracle.pow_steps(b, t) == np.float32(np.float32(oracle.pow_steps(b, t - 1)) * np.float32(b))


def test_oadam_constant_gradient_gives_unit_steps():
    """A constant gradient q: with bias correction m_hat_t = q and
    v_hat_t = q^2 exactly at every t (the corrections undo the zero start),
    so u_t = sign(q) and w_t = w_{t-1} - alpha sign(q) after the first step.
    Powers of two for q and dyadic b1, b2 keep every operation exact."""
    d, T = 64, 9
    r = rng(150)
    q = (np.where(r.random(d) < 0.5, -1.0, 1.0) * 2.0 ** r.integers(-12, 4, d)).astype(np.float32)
    st = oracle.OAdamState(d, oracle.OAdam(alpha=0.125, beta1=0.5, beta2=0.75, eps=0.0))
    w = np.zeros(d, np.float32)
    for t in range(1, T + 1):
        before = w.copy()
        st.update(t, q, w)
        assert np.array_equal(st.u, np.sign(q).astype(np.float32)), t
        step = np.float32(0.125) * (np.float32(2.0 if t == 1 else 1.0) * np.sign(q)).astype(np.float32)
        assert np.array_equal(w, (before - step).astype(np.float32)), t
