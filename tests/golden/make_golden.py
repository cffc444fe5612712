"""Writes algorithm2_tiny.json: three steps of Algorithm 2 (DQGAN) on a tiny
problem for each compressor, computed by the fp32 oracle and checked, before
anything is written, against the exact rational replay (the inputs are
dyadic, so every fp32 operation of the method is exact here and the two
must agree to the bit; for the quantiser, whose levels r/7 and reciprocal
7/s are rounded in fp32, within 1e-6 of the scale).  Calls only
``oracle``.

    python tests/golden/make_golden.py

Cited definitions: Algorithm 2 (worker error feedback p = eta F + e,
residual e = p - Q(p), server average and update); Section 2.4 (scaled
sign, top-k, the b-bit stochastic quantiser of Hou et al.); Theorem 1
(top-k), the proof of Theorem 2 (quantiser levels).
"""
from __future__ import annotations

import json
import os
import sys
from fractions import Fraction

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))

import oracle  # noqa: E402
from oracle import exact  # noqa: E402

D, M, T, BUCKET, LR, SEED = 40, 2, 3, 32, 0.25, 12345
CASES = {
    "sign": dict(compressor=oracle.SIGN, bucket=BUCKET),
    "topk": dict(compressor=oracle.TOPK, k=5),
    "squant_b4": dict(compressor=oracle.SQUANT, bucket=BUCKET, bits=4),
    "identity": dict(compressor=oracle.IDENTITY),
}


def gradients():
    """Dyadic gradients: integers in [-32, 32] / 16, seeded."""
    rng = np.random.default_rng(SEED)
    return (rng.integers(-32, 33, size=(T, M, D)) / 16.0).astype(np.float32)


def hexf(a) -> list:
    return [f"{int(x):08x}" for x in np.ascontiguousarray(a, np.float32).view(np.uint32)]


def exact_compressor(name, cfg):
    if name == "sign":
        return lambda p, m, t: exact.q_sign(p, BUCKET)
    if name == "topk":
        return lambda p, m, t: exact.q_topk(p, cfg.k)
    if name == "identity":
        return lambda p, m, t: exact.q_identity(p)

    def q(p, m, t):
        u = [Fraction(float(oracle.squant_uniform(SEED, m, t, j))) for j in range(D)]
        return exact.q_squant(p, BUCKET, 4, u)
    return q


def main():
    g = gradients()
    w0 = (np.arange(D, dtype=np.float32) - 20) / np.float32(64)
    out = {"about": __doc__.strip().splitlines()[0], "d": D, "M": M, "steps": T, "lr": LR, "seed": SEED,
           "gradients_f32_hex": [[hexf(g[t, m]) for m in range(M)] for t in range(T)],
           "w0_f32_hex": hexf(w0), "cases": {}}
    for name, kw in CASES.items():
        cfg = oracle.Config(d=D, M=M, lr=LR, seed=SEED, **kw)
        st = oracle.State(cfg)
        w = w0.copy()
        ex = exact.ExactDQGAN(exact.frac_vec(w0), M, Fraction(LR), exact_compressor(name, cfg))
        steps = []
        for t in range(T):
            msgs = st.step(g[t], w)
            ex.step(lambda m, tt, wh: exact.frac_vec(g[tt - 1, m]))
            # the fp32 oracle equals the exact replay on these inputs
            w_ex = np.array([float(x) for x in ex.w], np.float64)
            if name == "squant_b4":
                assert np.max(np.abs(w - w_ex)) <= 1e-6 * max(1.0, np.max(np.abs(w_ex))), (name, t)
            else:
                assert np.array_equal(w, w_ex.astype(np.float32)), (name, t)
                for m in range(M):
                    e_ex = np.array([float(x) for x in ex.e[m]], np.float32)
                    assert np.array_equal(st.e[m], e_ex), (name, t, m)
            steps.append({"messages_hex": [msgs[m].tobytes().hex() for m in range(M)],
                          "e_f32_hex": [hexf(st.e[m]) for m in range(M)],
                          "w_f32_hex": hexf(w)})
        out["cases"][name] = {"config": {k: int(v) for k, v in kw.items()}, "steps": steps}
    path = os.path.join(HERE, "algorithm2_tiny.json")
    with open(path, "w") as f:
        json.dump(out, f, indent=1)
    print(path)


if __name__ == "__main__":
    main()
