"""Helpers shared by the GPU parity tests: run the CUDA path through the C-ABI
and the oracle side by side on identical seeded inputs, and compare.

Comparison rules (the tolerances are written here, once):

* packed messages (sign words, quantisation codes, top-k records, scales)
  and the residuals e and lookahead offsets h are compared bit for bit:
  both sides form p, the scales and Q(p) with the same rounded fp32
  operations in the same order;
* parameters w are compared bit for bit as well: both sides sum the M
  decoded messages in the one order the library and the oracle fix (the M
  values padded with +0 to a power of two, summed pairwise).  The stated
  fp32 tolerance -- max relative error 1e-5 per step and 1e-4 after a whole
  run, per element, relative to max(|y_j|, 1e-6 max_j |y_j|) -- is checked
  first, so that a failure reports how far apart the values are.
"""
from __future__ import annotations

import numpy as np

import oracle

STEP_RTOL = 1e-5
RUN_RTOL = 1e-4
FLOOR = 1e-6


def rel_err(x: np.ndarray, y: np.ndarray) -> float:
    """max_j |x_j - y_j| / max(|y_j|, FLOOR * max_j |y_j|), 0 for empty input."""
    x = np.asarray(x, np.float64)
    y = np.asarray(y, np.float64)
    if y.size == 0:
        return 0.0
    floor = FLOOR * np.max(np.abs(y))
    denom = np.maximum(np.abs(y), floor)
    diff = np.abs(x - y)
    with np.errstate(divide="ignore", invalid="ignore"):
        r = np.where(diff == 0.0, 0.0, diff / np.where(denom == 0.0, 1.0, denom))
    r = np.where((denom == 0.0) & (diff != 0.0), np.inf, r)
    return float(np.max(r))


def assert_params_equal(got: np.ndarray, want: np.ndarray, ctx: str = "", rtol: float = STEP_RTOL):
    """w from the CUDA path against the oracle: within the per-element
    tolerance, then bit for bit."""
    err = rel_err(got, want)
    assert err <= rtol, f"{ctx}: params per-element rel err {err} > {rtol}"
    assert_bits_equal(got, want, f"{ctx}: params")


def sections(ocfg: oracle.Config, msg: np.ndarray) -> dict:
    """The meaningful bytes of a message, by name, as uint32 arrays."""
    off_s, off_p, total = oracle.layout(ocfg)
    d = ocfg.d
    msg = np.asarray(msg, np.uint8)
    if ocfg.compressor in (oracle.SIGN, oracle.SQUANT, oracle.QSGD):
        nb = len(oracle.bucket_starts(ocfg)) - 1
        nwords = -(-d // 32) if ocfg.compressor == oracle.SIGN else -(-d * ocfg.bits // 32)
        return {"scales": msg[off_s:off_s + 4 * nb].view(np.uint32),
                "payload": msg[off_p:off_p + 4 * nwords].view(np.uint32)}
    if ocfg.compressor == oracle.TOPK:
        return {"records": msg[:8 * ocfg.k].view(np.uint32)}
    return {"values": msg[:4 * d].view(np.uint32)}


def assert_messages_equal(ocfg: oracle.Config, got: np.ndarray, want: np.ndarray, ctx: str = ""):
    a, b = sections(ocfg, got), sections(ocfg, want)
    for name in b:
        if not np.array_equal(a[name], b[name]):
            bad = np.flatnonzero(a[name] != b[name])
            raise AssertionError(f"{ctx}: message section {name} differs at {bad.size} words, "
                                 f"first {bad[:5].tolist()}: gpu {a[name][bad[:5]].tolist()} "
                                 f"oracle {b[name][bad[:5]].tolist()}")


def assert_bits_equal(got: np.ndarray, want: np.ndarray, ctx: str = ""):
    g = np.ascontiguousarray(got, np.float32).view(np.uint32)
    w = np.ascontiguousarray(want, np.float32).view(np.uint32)
    if not np.array_equal(g, w):
        bad = np.flatnonzero(g != w)
        raise AssertionError(f"{ctx}: {bad.size} elements differ, first {bad[:5].tolist()}: "
                             f"gpu {got[bad[:5]].tolist()} oracle {want[bad[:5]].tolist()}")


def oracle_config(d, M, compressor, lr=1e-3, bucket=512, k=1, bits=8, seed=0, keep=False, segments=None):
    return oracle.Config(d=d, M=M, compressor=compressor, lr=lr, bucket=bucket, k=k, bits=bits,
                         seed=seed, keep_lookahead=keep, segments=segments)


def slice_messages(ocfg: oracle.Config, msgs: np.ndarray, a: int, b: int):
    """Sub-messages covering elements [a, b), where a and b are bucket starts
    (or b = d), and the matching oracle config (layer segments clipped to the
    range), so the oracle server can be run on a slice of a full-size
    problem.  Pure byte slicing: no arithmetic of the method."""
    assert ocfg.compressor in (oracle.SIGN, oracle.SQUANT, oracle.QSGD)
    starts = oracle.bucket_starts(ocfg)
    b0 = int(np.searchsorted(starts, a))
    b1 = int(np.searchsorted(starts, b)) if b < ocfg.d else len(starts) - 1
    assert starts[b0] == a and (b == ocfg.d or starts[b1] == b), "slice ends must be bucket starts"
    segs = None
    if ocfg.segments is not None:
        inner = [int(x) - a for x in ocfg.segments if a < x < b]
        segs = tuple([0] + inner + [b - a])
    sub = oracle.Config(d=b - a, M=ocfg.M, compressor=ocfg.compressor, lr=ocfg.lr, bucket=ocfg.bucket,
                        k=ocfg.k, bits=ocfg.bits, seed=ocfg.seed, segments=segs)
    off_s, off_p, _ = oracle.layout(ocfg)
    s_off_s, s_off_p, s_total = oracle.layout(sub)
    bits = 1 if ocfg.compressor == oracle.SIGN else ocfg.bits
    assert (a * bits) % 32 == 0
    out = np.zeros((ocfg.M, s_total), np.uint8)
    w0, w1 = a * bits // 32, -(-(b * bits) // 32)
    for m in range(ocfg.M):
        out[m, s_off_s:s_off_s + 4 * (b1 - b0)] = msgs[m, off_s + 4 * b0:off_s + 4 * b1]
        out[m, s_off_p:s_off_p + 4 * (w1 - w0)] = msgs[m, off_p + 4 * w0:off_p + 4 * w1]
    return sub, out
