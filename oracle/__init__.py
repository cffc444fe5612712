"""DQGAN oracle -- TEST INFRASTRUCTURE ONLY.

Python access (ctypes + numpy) to the plain C statement of Algorithm 2 in
``dqgan_oracle.c`` and to the exact-rational replay in ``exact.py``.  Only the
tests, ``__graft_entry__.smoke()`` and the CPU-baseline leg of ``bench.py``
may import this package; the product path never does.

Conventions (restated, not shared, with the CUDA library):

* compressors: 0 scaled sign, 1 top-k, 2 b-bit stochastic quantiser with
  the l_inf scale (Hou et al.), 3 identity, 4 b-bit stochastic quantiser
  with the l2 scale (QSGD);
* arrays are numpy ``float32`` (gradients, residuals, parameters) and
  ``uint8`` (messages);
* ``step`` is the iteration index t of Algorithm 2, starting at 1.
"""
from __future__ import annotations

import ctypes
import dataclasses

import numpy as np

from .build_oracle import build_oracle

SIGN, TOPK, SQUANT, IDENTITY, QSGD = 0, 1, 2, 3, 4
COMPRESSOR_NAMES = {"sign": SIGN, "topk": TOPK, "squant": SQUANT, "identity": IDENTITY, "qsgd": QSGD}


class _OrcCfg(ctypes.Structure):
    _fields_ = [
        ("d", ctypes.c_int64),
        ("k", ctypes.c_int64),
        ("lr", ctypes.c_float),
        ("M", ctypes.c_int32),
        ("compressor", ctypes.c_int32),
        ("bucket", ctypes.c_int32),
        ("bits", ctypes.c_int32),
        ("keep_lookahead", ctypes.c_int32),
        ("seed", ctypes.c_uint64),
        ("nseg", ctypes.c_int32),
        ("seg", ctypes.POINTER(ctypes.c_int64)),
    ]


class _OrcOAdam(ctypes.Structure):
    _fields_ = [
        ("alpha", ctypes.c_float),
        ("beta1", ctypes.c_float),
        ("beta2", ctypes.c_float),
        ("eps", ctypes.c_float),
        ("adaptive", ctypes.c_int32),
        ("bias_correction", ctypes.c_int32),
    ]


@dataclasses.dataclass
class OAdam:
    """Optimistic Adam server update (see orc_oadam_update)."""
    alpha: float = 1e-3
    beta1: float = 0.5
    beta2: float = 0.999
    eps: float = 1e-8
    adaptive: bool = True
    bias_correction: bool = True

    def c_struct(self) -> _OrcOAdam:
        return _OrcOAdam(alpha=self.alpha, beta1=self.beta1, beta2=self.beta2, eps=self.eps,
                         adaptive=1 if self.adaptive else 0, bias_correction=1 if self.bias_correction else 0)


@dataclasses.dataclass
class Config:
    d: int
    M: int
    compressor: int
    lr: float = 1e-3
    bucket: int = 512
    k: int = 1
    bits: int = 8
    seed: int = 0
    keep_lookahead: bool = False
    segments: tuple | None = None  # layer segment offsets 0 = s_0 < ... < s_n = d, or None

    def c_struct(self) -> _OrcCfg:
        c = _OrcCfg(d=self.d, k=self.k, lr=self.lr, M=self.M, compressor=self.compressor,
                    bucket=self.bucket, bits=self.bits,
                    keep_lookahead=1 if self.keep_lookahead else 0, seed=self.seed)
        if self.segments is not None:
            offs = np.ascontiguousarray(self.segments, dtype=np.int64)
            assert offs.ndim == 1 and offs.size >= 2 and offs[0] == 0 and offs[-1] == self.d
            assert np.all(np.diff(offs) > 0)
            c.nseg = offs.size - 1
            c.seg = offs.ctypes.data_as(ctypes.POINTER(ctypes.c_int64))
            c._keep = offs  # the offsets must outlive the struct
        return c


_lib = None


def lib() -> ctypes.CDLL:
    global _lib
    if _lib is None:
        path = build_oracle()
        L = ctypes.CDLL(path)
        P = ctypes.POINTER
        f32p, u8p = P(ctypes.c_float), P(ctypes.c_uint8)
        cfgp = P(_OrcCfg)
        L.orc_philox4x32_10.argtypes = [P(ctypes.c_uint32), P(ctypes.c_uint32), P(ctypes.c_uint32)]
        L.orc_philox4x32_10.restype = None
        L.orc_squant_uniform.argtypes = [ctypes.c_uint64, ctypes.c_int32, ctypes.c_int64, ctypes.c_int64]
        L.orc_squant_uniform.restype = ctypes.c_float
        L.orc_layout.argtypes = [cfgp, P(ctypes.c_int64), P(ctypes.c_int64)]
        L.orc_layout.restype = ctypes.c_int64
        L.orc_sign_l1.argtypes = [f32p, ctypes.c_int64, ctypes.c_int32]
        L.orc_sign_l1.restype = ctypes.c_float
        L.orc_sign_scale.argtypes = [f32p, ctypes.c_int64, ctypes.c_int32]
        L.orc_sign_scale.restype = ctypes.c_float
        L.orc_qsgd_sumsq.argtypes = [f32p, ctypes.c_int64, ctypes.c_int32]
        L.orc_qsgd_sumsq.restype = ctypes.c_float
        L.orc_qsgd_scale.argtypes = [f32p, ctypes.c_int64, ctypes.c_int32]
        L.orc_qsgd_scale.restype = ctypes.c_float
        L.orc_squant_decode.argtypes = [ctypes.c_int32, ctypes.c_float, ctypes.c_int32]
        L.orc_squant_decode.restype = ctypes.c_float
        L.orc_topk_select.argtypes = [f32p, ctypes.c_int64, ctypes.c_int64, u8p]
        L.orc_topk_select.restype = None
        L.orc_decode.argtypes = [cfgp, u8p, f32p]
        L.orc_decode.restype = None
        L.orc_worker_step.argtypes = [cfgp, ctypes.c_int32, ctypes.c_int64, f32p, f32p, f32p, u8p]
        L.orc_worker_step.restype = None
        L.orc_pairwise_sum.argtypes = [f32p, ctypes.c_int32]
        L.orc_pairwise_sum.restype = ctypes.c_float
        L.orc_server_step.argtypes = [cfgp, u8p, ctypes.c_int64, f32p]
        L.orc_server_step.restype = None
        L.orc_server_step_range.argtypes = [cfgp, u8p, ctypes.c_int64, f32p, ctypes.c_int64, ctypes.c_int64]
        L.orc_server_step_range.restype = None
        L.orc_server_average_range.argtypes = [cfgp, u8p, ctypes.c_int64, f32p, ctypes.c_int64, ctypes.c_int64]
        L.orc_server_average_range.restype = None
        L.orc_pow_steps.argtypes = [ctypes.c_float, ctypes.c_int64]
        L.orc_pow_steps.restype = ctypes.c_float
        oap = P(_OrcOAdam)
        L.orc_oadam_update.argtypes = [oap, ctypes.c_int64, ctypes.c_int64, f32p, f32p, f32p, f32p, f32p]
        L.orc_oadam_update.restype = None
        L.orc_server_step_oadam_range.argtypes = [cfgp, u8p, ctypes.c_int64, oap, ctypes.c_int64, f32p, f32p,
                                                  f32p, f32p, ctypes.c_int64, ctypes.c_int64]
        L.orc_server_step_oadam_range.restype = None
        L.orc_lookahead.argtypes = [ctypes.c_int64, f32p, f32p, f32p]
        L.orc_lookahead.restype = None
        L.orc_bucket_count.argtypes = [cfgp]
        L.orc_bucket_count.restype = ctypes.c_int64
        L.orc_bucket_starts.argtypes = [cfgp, P(ctypes.c_int64)]
        L.orc_bucket_starts.restype = None
        _lib = L
    return _lib


def _f32(a: np.ndarray):
    assert a.dtype == np.float32 and a.flags.c_contiguous
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_float))


def _u8(a: np.ndarray):
    assert a.dtype == np.uint8 and a.flags.c_contiguous
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_uint8))


def philox4x32_10(ctr, key) -> np.ndarray:
    c = (ctypes.c_uint32 * 4)(*[int(x) & 0xFFFFFFFF for x in ctr])
    k = (ctypes.c_uint32 * 2)(*[int(x) & 0xFFFFFFFF for x in key])
    o = (ctypes.c_uint32 * 4)()
    lib().orc_philox4x32_10(c, k, o)
    return np.array(list(o), dtype=np.uint32)


def squant_uniform(seed: int, worker: int, step: int, j: int) -> float:
    return float(lib().orc_squant_uniform(seed, worker, step, j))


def layout(cfg: Config):
    """(scales offset, payload offset, total bytes) of one message."""
    a, b = ctypes.c_int64(), ctypes.c_int64()
    total = lib().orc_layout(ctypes.byref(cfg.c_struct()), ctypes.byref(a), ctypes.byref(b))
    return a.value, b.value, total


def message_bytes(cfg: Config) -> int:
    return layout(cfg)[2]


def bucket_starts(cfg: Config) -> np.ndarray:
    """starts[0..nb]: bucket b covers [starts[b], starts[b+1])."""
    c = cfg.c_struct()
    nb = lib().orc_bucket_count(ctypes.byref(c))
    out = np.zeros(nb + 1, dtype=np.int64)
    lib().orc_bucket_starts(ctypes.byref(c), out.ctypes.data_as(ctypes.POINTER(ctypes.c_int64)))
    return out


def sign_l1(x: np.ndarray, bucket: int) -> float:
    x = np.ascontiguousarray(x, dtype=np.float32)
    return float(lib().orc_sign_l1(_f32(x), x.size, bucket))


def sign_scale(x: np.ndarray, bucket: int) -> float:
    x = np.ascontiguousarray(x, dtype=np.float32)
    return float(lib().orc_sign_scale(_f32(x), x.size, bucket))


def qsgd_sumsq(x: np.ndarray, bucket: int) -> float:
    x = np.ascontiguousarray(x, dtype=np.float32)
    return float(lib().orc_qsgd_sumsq(_f32(x), x.size, bucket))


def qsgd_scale(x: np.ndarray, bucket: int) -> float:
    x = np.ascontiguousarray(x, dtype=np.float32)
    return float(lib().orc_qsgd_scale(_f32(x), x.size, bucket))


def squant_decode(code: int, s: float, K: int) -> float:
    return float(lib().orc_squant_decode(code, s, K))


def topk_select(p: np.ndarray, k: int) -> np.ndarray:
    p = np.ascontiguousarray(p, dtype=np.float32)
    sel = np.zeros(p.size, dtype=np.uint8)
    lib().orc_topk_select(_f32(p), p.size, k, _u8(sel))
    return sel.astype(bool)


def decode(cfg: Config, msg: np.ndarray) -> np.ndarray:
    q = np.zeros(cfg.d, dtype=np.float32)
    lib().orc_decode(ctypes.byref(cfg.c_struct()), _u8(np.ascontiguousarray(msg)), _f32(q))
    return q


def worker_step(cfg: Config, worker: int, step: int, g: np.ndarray, e: np.ndarray,
                h: np.ndarray | None = None) -> np.ndarray:
    """One worker step of Algorithm 2; updates e (and h) in place, returns the message."""
    g = np.ascontiguousarray(g, dtype=np.float32)
    msg = np.zeros(message_bytes(cfg), dtype=np.uint8)
    hp = _f32(h) if h is not None else ctypes.POINTER(ctypes.c_float)()
    lib().orc_worker_step(ctypes.byref(cfg.c_struct()), worker, step, _f32(g), _f32(e), hp, _u8(msg))
    return msg


def pairwise_sum(values) -> float:
    """The server's fixed-order sum of M values (padded with +0 to a power of two, summed pairwise)."""
    v = np.ascontiguousarray(values, dtype=np.float32)
    M = v.size
    P = 1
    while P < M:
        P *= 2
    buf = np.zeros(P, dtype=np.float32)
    buf[:M] = v
    return float(lib().orc_pairwise_sum(_f32(buf), M))


def server_step(cfg: Config, msgs: np.ndarray, w: np.ndarray) -> None:
    """Server step of Algorithm 2 on M stacked messages (M x message_bytes); updates w."""
    msgs = np.ascontiguousarray(msgs, dtype=np.uint8)
    assert msgs.ndim == 2 and msgs.shape[0] == cfg.M
    lib().orc_server_step(ctypes.byref(cfg.c_struct()), _u8(msgs), msgs.shape[1], _f32(w))


def server_step_range(cfg: Config, msgs: np.ndarray, w: np.ndarray, j0: int, j1: int) -> None:
    """The server step on elements [j0, j1) of w only (disjoint ranges may run in parallel threads)."""
    assert msgs.dtype == np.uint8 and msgs.flags.c_contiguous and msgs.ndim == 2 and msgs.shape[0] == cfg.M
    assert 0 <= j0 <= j1 <= cfg.d and w.size == cfg.d
    lib().orc_server_step_range(ctypes.byref(cfg.c_struct()), _u8(msgs), msgs.shape[1], _f32(w), j0, j1)


def server_average(cfg: Config, msgs: np.ndarray, j0: int = 0, j1: int | None = None) -> np.ndarray:
    """q_hat = (1/M) sum_m Q_m for elements [j0, j1) (the server's fixed-order average)."""
    j1 = cfg.d if j1 is None else j1
    msgs = np.ascontiguousarray(msgs, dtype=np.uint8)
    out = np.zeros(max(j1 - j0, 1), np.float32)
    lib().orc_server_average_range(ctypes.byref(cfg.c_struct()), _u8(msgs), msgs.shape[1], _f32(out), j0, j1)
    return out[:j1 - j0]


def pow_steps(b: float, t: int) -> float:
    return float(lib().orc_pow_steps(b, t))


class OAdamState:
    """The server's Optimistic Adam state for d parameters: m, v, u_prev (zero at the start)."""

    def __init__(self, d: int, opt: OAdam):
        self.opt = opt
        self.m = np.zeros(d, np.float32)
        self.v = np.zeros(d, np.float32)
        self.u = np.zeros(d, np.float32)

    def update(self, t: int, q_hat: np.ndarray, w: np.ndarray) -> None:
        """One Optimistic Adam step at iteration t on w (in place) from the averaged update q_hat."""
        q_hat = np.ascontiguousarray(q_hat, dtype=np.float32)
        c = self.opt.c_struct()
        lib().orc_oadam_update(ctypes.byref(c), t, w.size, _f32(q_hat), _f32(self.m), _f32(self.v), _f32(self.u),
                               _f32(w))

    def server_step_range(self, cfg: Config, t: int, msgs: np.ndarray, w: np.ndarray, j0: int, j1: int) -> None:
        """Server step of Algorithm 2 with the Optimistic Adam update, on elements [j0, j1)."""
        msgs = np.ascontiguousarray(msgs, dtype=np.uint8)
        c = self.opt.c_struct()
        lib().orc_server_step_oadam_range(ctypes.byref(cfg.c_struct()), _u8(msgs), msgs.shape[1], ctypes.byref(c), t,
                                          _f32(self.m), _f32(self.v), _f32(self.u), _f32(w), j0, j1)


def lookahead(w: np.ndarray, h: np.ndarray) -> np.ndarray:
    out = np.empty_like(w)
    lib().orc_lookahead(w.size, _f32(w), _f32(h), _f32(out))
    return out


class State:
    """Oracle state of Algorithm 2 for M workers: residuals e, lookahead offsets h, step t."""

    def __init__(self, cfg: Config):
        self.cfg = cfg
        self.e = np.zeros((cfg.M, cfg.d), dtype=np.float32)
        self.h = np.zeros((cfg.M, cfg.d), dtype=np.float32) if cfg.keep_lookahead else None
        self.t = 1

    def compress_all(self, g: np.ndarray, workers=None) -> np.ndarray:
        """Worker steps for all (or the listed) workers at the current step."""
        cfg = self.cfg
        ws = range(cfg.M) if workers is None else workers
        msgs = np.zeros((cfg.M, message_bytes(cfg)), dtype=np.uint8)
        for i in ws:
            e_i = self.e[i]
            h_i = self.h[i] if self.h is not None else None
            msgs[i] = worker_step(cfg, i, self.t, g[i], e_i, h_i)
        return msgs

    def server(self, msgs: np.ndarray, w: np.ndarray) -> None:
        server_step(self.cfg, msgs, w)
        self.t += 1

    def step(self, g: np.ndarray, w: np.ndarray) -> np.ndarray:
        msgs = self.compress_all(g)
        self.server(msgs, w)
        return msgs
