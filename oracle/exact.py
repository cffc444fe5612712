"""Exact-rational replay of Algorithm 2 -- TEST INFRASTRUCTURE ONLY.

Every quantity is a ``fractions.Fraction``; nothing is rounded.  This is the
method as the paper states it in real arithmetic, used on tiny problems
(d <= 16, M <= 4) to pin the fp32 oracle and to check the paper's identities
exactly:

* Algorithm 2 (DQGAN): lookahead, p = eta*F + e, p_hat = Q(p), e = p - p_hat,
  q_hat = mean of the p_hat, w = w - q_hat;
* compressors of Section 2.4 / Section 3.2 (scaled sign with the l1 mean
  scale, top-k of Theorem 1, the b-bit stochastic quantiser of the proof of
  Theorem 2 with the l_inf scale and uniform levels);
* the stochastic quantiser takes its uniform draws as inputs, so a replay can
  use the very draws the fp32 oracle made.

Lists of Fractions stand for vectors.
"""
from __future__ import annotations

from fractions import Fraction
from typing import Callable, Sequence

Vec = list  # list[Fraction]


def frac_vec(xs) -> Vec:
    return [Fraction(float(x)) if not isinstance(x, Fraction) else x for x in xs]


def sq_norm(v: Sequence[Fraction]) -> Fraction:
    return sum((x * x for x in v), Fraction(0))


def l1(v: Sequence[Fraction]) -> Fraction:
    return sum((abs(x) for x in v), Fraction(0))


# --- compressors -----------------------------------------------------------

def q_sign(p: Vec, bucket: int) -> Vec:
    """Scaled sign per bucket: q_j = -s if p_j < 0 else s, s = ||p_b||_1 / n_b."""
    out = []
    for start in range(0, len(p), bucket):
        blk = p[start:start + bucket]
        s = l1(blk) / len(blk)
        out.extend(-s if x < 0 else s for x in blk)
    return out


def q_topk(p: Vec, k: int) -> Vec:
    """Keep the k entries of largest |p_j|, ties to the lower index."""
    order = sorted(range(len(p)), key=lambda j: (-abs(p[j]), j))
    keep = set(order[:k])
    return [p[j] if j in keep else Fraction(0) for j in range(len(p))]


def q_squant(p: Vec, bucket: int, bits: int, uniforms: Sequence[Fraction], scales=None) -> Vec:
    """b-bit stochastic quantiser, s = max |p| per bucket (or the given
    per-bucket scales, e.g. QSGD's l2 norms), levels B_r = r/K.

    Element j rounds |p_j|/s * K up from level r = floor(.) with the draw
    uniforms[j]: up iff u < frac(|p_j| K / s)."""
    K = 2 ** (bits - 1) - 1
    out = []
    for bi, start in enumerate(range(0, len(p), bucket)):
        blk = p[start:start + bucket]
        s = max((abs(x) for x in blk), default=Fraction(0)) if scales is None else scales[bi]
        for off, x in enumerate(blk):
            if s == 0:
                out.append(Fraction(0))
                continue
            t = abs(x) * K / s
            r = t.numerator // t.denominator
            f = t - r
            level = r + (1 if uniforms[start + off] < f else 0)
            level = min(level, K)
            mag = s * Fraction(level, K)
            out.append(-mag if x < 0 else mag)
    return out


def q_identity(p: Vec) -> Vec:
    return list(p)


# --- Algorithm 2 ------------------------------------------------------------

class ExactDQGAN:
    """Algorithm 2 on M workers in exact arithmetic.

    ``compress(p, worker, step)`` is the compressor Q; ``grad(m, t, w_half)``
    returns the worker's stochastic gradient F(w_half; xi_t^(m)).
    """

    def __init__(self, w0: Vec, M: int, lr: Fraction, compress: Callable[[Vec, int, int], Vec]):
        self.w = list(w0)
        self.M = M
        self.lr = Fraction(lr)
        self.compress = compress
        d = len(w0)
        self.e = [[Fraction(0)] * d for _ in range(M)]
        self.F_prev = [[Fraction(0)] * d for _ in range(M)]  # F(w_{-3/2}) := 0 at t = 1
        self.t = 0
        self.history = []  # per step: dict of w_half, p, p_hat, e, q_hat, w

    def lookahead(self, m: int) -> Vec:
        """w_{t-1/2}^(m) = w_{t-1} - [eta F(w_{t-3/2}^(m)) + e_{t-1}^(m)]."""
        return [w - (self.lr * f + e) for w, f, e in zip(self.w, self.F_prev[m], self.e[m])]

    def step(self, grad: Callable[[int, int, Vec], Vec]) -> dict:
        self.t += 1
        t = self.t
        d = len(self.w)
        rec = {"w_half": [], "F": [], "p": [], "p_hat": [], "e": []}
        p_hats = []
        for m in range(self.M):
            w_half = self.lookahead(m)
            F = grad(m, t, w_half)
            p = [self.lr * f + e for f, e in zip(F, self.e[m])]
            p_hat = self.compress(p, m, t)
            self.e[m] = [a - b for a, b in zip(p, p_hat)]
            self.F_prev[m] = list(F)
            p_hats.append(p_hat)
            for key, val in (("w_half", w_half), ("F", F), ("p", p), ("p_hat", p_hat),
                             ("e", self.e[m])):
                rec[key].append(val)
        q_hat = [sum((p_hats[m][j] for m in range(self.M)), Fraction(0)) / self.M
                 for j in range(d)]
        self.w = [w - q for w, q in zip(self.w, q_hat)]
        rec["q_hat"] = q_hat
        rec["w"] = list(self.w)
        self.history.append(rec)
        return rec


# --- Optimistic Adam server update (the CPOAdam family of Section 4) --------

def exact_sqrt(x: Fraction) -> Fraction:
    """The square root of x when it is rational (x a square of a rational); else ValueError."""
    from math import isqrt
    if x < 0:
        raise ValueError("negative")
    n, d = x.numerator, x.denominator
    rn, rd = isqrt(n), isqrt(d)
    if rn * rn != n or rd * rd != d:
        raise ValueError("not a rational square")
    return Fraction(rn, rd)


class ExactOAdam:
    """Optimistic Adam (Daskalakis et al., ICLR 2018) on the server's
    averaged update, in exact arithmetic:
    m = b1 m + (1 - b1) q; v = b2 v + (1 - b2) q^2; with bias correction
    m_hat = m / (1 - b1^t), v_hat = v / (1 - b2^t); adaptive:
    u = m_hat / (sqrt(v_hat) + eps) (u = 0 where m_hat = 0), else u = m_hat;
    w = w - alpha (2 u - u_prev).  The square root must be rational (for
    example b2 = 0, where sqrt(v_hat) = |q|)."""

    def __init__(self, d: int, alpha, beta1, beta2, eps, adaptive: bool = True, bias_correction: bool = True):
        self.alpha, self.b1, self.b2, self.eps = (Fraction(x) for x in (alpha, beta1, beta2, eps))
        self.adaptive, self.bc = adaptive, bias_correction
        self.m = [Fraction(0)] * d
        self.v = [Fraction(0)] * d
        self.u = [Fraction(0)] * d

    def update(self, t: int, q_hat: Vec, w: Vec) -> Vec:
        c1 = 1 - self.b1 ** t if self.bc else Fraction(1)
        c2 = 1 - self.b2 ** t if self.bc else Fraction(1)
        out = []
        for j, (g, x) in enumerate(zip(q_hat, w)):
            self.m[j] = self.b1 * self.m[j] + (1 - self.b1) * g
            self.v[j] = self.b2 * self.v[j] + (1 - self.b2) * g * g
            mh, vh = self.m[j] / c1, self.v[j] / c2
            if self.adaptive:
                u = Fraction(0) if mh == 0 else mh / (exact_sqrt(vh) + self.eps)
            else:
                u = mh
            out.append(x - self.alpha * (2 * u - self.u[j]))
            self.u[j] = u
        return out
