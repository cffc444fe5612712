"""Thin Python binding of the DQGAN C-ABI (include/dqgan.h).

Argument marshalling only: every call goes straight to ``libdqgan.so``,
where every step of the hot path runs as a CUDA kernel.  Pointer arguments
accept a ``torch.Tensor`` (its ``data_ptr()``), a plain integer address, or
(for the host-copy calls) a numpy array.  There is no fallback: if the
library is missing, loading fails with an error.
"""
from __future__ import annotations

import ctypes
import os

HERE = os.path.dirname(os.path.abspath(__file__))
# The library to load: libdqgan.so next to this file, or the path the
# environment variable DQGAN_LIBRARY names (the checked build, for instance).
LIBRARY = os.environ.get("DQGAN_LIBRARY") or os.path.join(HERE, "libdqgan.so")

OK = 0
ERR_INVALID_ARG = -1
ERR_OOM = -2
ERR_CUDA = -3
ERR_UNSUPPORTED = -4
ERR_TIMEOUT = -5
ERR_BOUNDS = -6

SIGN, TOPK, SQUANT, IDENTITY, QSGD = 0, 1, 2, 3, 4
KEEP_LOOKAHEAD = 1


class DqganError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"dqgan status {status}: {message}")
        self.status = status


class Config(ctypes.Structure):
    """Mirror of ``dqgan_config`` (56 bytes, no padding)."""
    _fields_ = [
        ("d", ctypes.c_int64),
        ("k", ctypes.c_int64),
        ("lr", ctypes.c_float),
        ("M", ctypes.c_int32),
        ("compressor", ctypes.c_int32),
        ("bucket", ctypes.c_int32),
        ("bits", ctypes.c_int32),
        ("flags", ctypes.c_uint32),
        ("seed", ctypes.c_uint64),
        ("cuda_stream", ctypes.c_void_p),
    ]


assert ctypes.sizeof(Config) == 56

SERVER_OMD, SERVER_OADAM = 0, 1
OADAM_ADAPTIVE, OADAM_BIAS_CORRECTION = 1, 2


class ServerOptimizer(ctypes.Structure):
    """Mirror of ``dqgan_server_optimizer`` (28 bytes, no padding)."""
    _fields_ = [
        ("kind", ctypes.c_int32),
        ("flags", ctypes.c_uint32),
        ("alpha", ctypes.c_float),
        ("beta1", ctypes.c_float),
        ("beta2", ctypes.c_float),
        ("eps", ctypes.c_float),
        ("reserved", ctypes.c_uint32),
    ]


assert ctypes.sizeof(ServerOptimizer) == 28


def oadam(alpha: float, beta1: float, beta2: float, eps: float, adaptive: bool = True,
          bias_correction: bool = True) -> ServerOptimizer:
    flags = (OADAM_ADAPTIVE if adaptive else 0) | (OADAM_BIAS_CORRECTION if bias_correction else 0)
    return ServerOptimizer(kind=SERVER_OADAM, flags=flags, alpha=alpha, beta1=beta1, beta2=beta2, eps=eps)

_lib = None


def load_library(path: str = LIBRARY) -> ctypes.CDLL:
    """Load libdqgan.so (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is missing: build the CUDA library first "
                           "(python -m paper_2010_13359_gb300.build)")
    L = ctypes.CDLL(path)
    H = ctypes.c_void_p
    P = ctypes.c_void_p
    i32, i64, u64 = ctypes.c_int32, ctypes.c_int64, ctypes.c_uint64
    cfgp = ctypes.POINTER(Config)
    sig = {
        "dqgan_message_layout": (ctypes.c_int, [cfgp, ctypes.POINTER(i64), ctypes.POINTER(i64),
                                                ctypes.POINTER(i64)]),
        "dqgan_validate_config": (ctypes.c_int, [cfgp]),
        "dqgan_create": (ctypes.c_int, [cfgp, ctypes.POINTER(H)]),
        "dqgan_destroy": (ctypes.c_int, [H]),
        "dqgan_message_bytes": (i64, [H]),
        "dqgan_worker_compress": (ctypes.c_int, [H, i32, P, P]),
        "dqgan_workers_compress_all": (ctypes.c_int, [H, P, i64, P]),
        "dqgan_server_aggregate_update": (ctypes.c_int, [H, P, P]),
        "dqgan_worker_lookahead": (ctypes.c_int, [H, i32, P, P]),
        "dqgan_synchronize": (ctypes.c_int, [H]),
        "dqgan_get_residual": (ctypes.c_int, [H, i32, P]),
        "dqgan_set_residual": (ctypes.c_int, [H, i32, P]),
        "dqgan_get_lookahead": (ctypes.c_int, [H, i32, P]),
        "dqgan_set_lookahead": (ctypes.c_int, [H, i32, P]),
        "dqgan_get_step": (i64, [H]),
        "dqgan_set_step": (ctypes.c_int, [H, i64]),
        "dqgan_state_bytes": (i64, [H]),
        "dqgan_save_state": (ctypes.c_int, [H, P, i64]),
        "dqgan_load_state": (ctypes.c_int, [H, P, i64]),
        "dqgan_launch_count": (u64, [H]),
        "dqgan_last_error": (ctypes.c_char_p, [H]),
        "dqgan_topk_compress_noalloc": (ctypes.c_int, [P, P, P, i64, i64, ctypes.c_float, P]),
        "dqgan_selftest_wait_timeout": (ctypes.c_int, [H, ctypes.c_uint32]),
        "dqgan_set_segments": (ctypes.c_int, [H, ctypes.POINTER(i64), i32]),
        "dqgan_set_server_optimizer": (ctypes.c_int, [H, ctypes.POINTER(ServerOptimizer)]),
        "dqgan_workers_compress_range": (ctypes.c_int, [H, i32, i32, P, i64, P]),
        "dqgan_set_local_workers": (ctypes.c_int, [H, i32, i32]),
        "dqgan_get_server_state": (ctypes.c_int, [H, i32, P]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(L, name)
        fn.restype = res
        fn.argtypes = args
    _lib = L
    return L


def _ptr(x) -> int | None:
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if hasattr(x, "data_ptr"):
        return x.data_ptr()
    if hasattr(x, "ctypes"):  # numpy
        return x.ctypes.data
    raise TypeError(f"cannot take a pointer of {type(x)}")


def make_config(d: int, M: int, compressor: int, lr: float = 1e-3, bucket: int = 512, k: int = 1,
                bits: int = 8, seed: int = 0, flags: int = 0, cuda_stream: int | None = None) -> Config:
    return Config(d=d, k=k, lr=lr, M=M, compressor=compressor, bucket=bucket, bits=bits, flags=flags,
                  seed=seed, cuda_stream=cuda_stream)


def _check(status: int, handle=None):
    if status != OK:
        msg = load_library().dqgan_last_error(handle)
        raise DqganError(status, msg.decode() if msg else "")


def message_layout(cfg: Config) -> tuple[int, int, int]:
    """(scales offset, payload offset, total bytes); host only."""
    a, b, c = ctypes.c_int64(), ctypes.c_int64(), ctypes.c_int64()
    _check(load_library().dqgan_message_layout(ctypes.byref(cfg), ctypes.byref(a), ctypes.byref(b),
                                               ctypes.byref(c)))
    return a.value, b.value, c.value


def validate_config(cfg: Config) -> None:
    _check(load_library().dqgan_validate_config(ctypes.byref(cfg)))


class Handle:
    """Owner of one ``dqgan_handle``; methods are the C-ABI calls of the same name."""

    def __init__(self, cfg: Config):
        self.cfg = cfg
        L = load_library()
        h = ctypes.c_void_p()
        _check(L.dqgan_create(ctypes.byref(cfg), ctypes.byref(h)))
        self._h = h

    # -- lifetime -------------------------------------------------------------
    def destroy(self) -> None:
        if self._h is not None and self._h.value:
            _check(load_library().dqgan_destroy(self._h))
        self._h = None

    def __del__(self):
        try:
            self.destroy()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.destroy()

    @property
    def raw(self) -> ctypes.c_void_p:
        return self._h

    # -- hot path -------------------------------------------------------------
    def set_segments(self, offsets) -> None:
        """dqgan_set_segments: per-layer buckets; offsets from 0 to d (None: flat)."""
        if offsets is None:
            _check(load_library().dqgan_set_segments(self._h, None, 0), self._h)
            return
        arr = (ctypes.c_int64 * len(offsets))(*[int(x) for x in offsets])
        _check(load_library().dqgan_set_segments(self._h, arr, len(offsets) - 1), self._h)

    def set_server_optimizer(self, opt: ServerOptimizer) -> None:
        _check(load_library().dqgan_set_server_optimizer(self._h, ctypes.byref(opt)), self._h)

    def get_server_state(self, which: int, dst) -> None:
        """which: 0 m, 1 v, 2 u_prev (d fp32 into dst, host or device)."""
        _check(load_library().dqgan_get_server_state(self._h, which, _ptr(dst)), self._h)

    def message_bytes(self) -> int:
        return int(load_library().dqgan_message_bytes(self._h))

    def worker_compress(self, i: int, g, out_msg) -> None:
        _check(load_library().dqgan_worker_compress(self._h, i, _ptr(g), _ptr(out_msg)), self._h)

    def workers_compress_all(self, g_all, g_stride: int, msgs_all) -> None:
        _check(load_library().dqgan_workers_compress_all(self._h, _ptr(g_all), g_stride, _ptr(msgs_all)),
               self._h)

    def workers_compress_range(self, first: int, count: int, g, g_stride: int, msgs) -> None:
        _check(load_library().dqgan_workers_compress_range(self._h, first, count, _ptr(g), g_stride, _ptr(msgs)),
               self._h)

    def set_local_workers(self, first: int, count: int) -> None:
        _check(load_library().dqgan_set_local_workers(self._h, first, count), self._h)

    def server_aggregate_update(self, msgs_all, params) -> None:
        _check(load_library().dqgan_server_aggregate_update(self._h, _ptr(msgs_all), _ptr(params)), self._h)

    def worker_lookahead(self, i: int, params, out_w_half) -> None:
        _check(load_library().dqgan_worker_lookahead(self._h, i, _ptr(params), _ptr(out_w_half)), self._h)

    def synchronize(self) -> None:
        _check(load_library().dqgan_synchronize(self._h), self._h)

    def selftest_wait_timeout(self, polls: int = 0) -> None:
        """Enqueue the bounded-wait self-test; the next synchronize() raises
        DqganError with status ERR_TIMEOUT."""
        _check(load_library().dqgan_selftest_wait_timeout(self._h, polls), self._h)

    # -- state ----------------------------------------------------------------
    def get_residual(self, i: int, dst) -> None:
        _check(load_library().dqgan_get_residual(self._h, i, _ptr(dst)), self._h)

    def set_residual(self, i: int, src) -> None:
        _check(load_library().dqgan_set_residual(self._h, i, _ptr(src)), self._h)

    def get_lookahead(self, i: int, dst) -> None:
        _check(load_library().dqgan_get_lookahead(self._h, i, _ptr(dst)), self._h)

    def set_lookahead(self, i: int, src) -> None:
        _check(load_library().dqgan_set_lookahead(self._h, i, _ptr(src)), self._h)

    def get_step(self) -> int:
        return int(load_library().dqgan_get_step(self._h))

    def set_step(self, t: int) -> None:
        _check(load_library().dqgan_set_step(self._h, t), self._h)

    def state_bytes(self) -> int:
        return int(load_library().dqgan_state_bytes(self._h))

    def save_state(self, host_dst, nbytes: int) -> None:
        _check(load_library().dqgan_save_state(self._h, _ptr(host_dst), nbytes), self._h)

    def load_state(self, host_src, nbytes: int) -> None:
        _check(load_library().dqgan_load_state(self._h, _ptr(host_src), nbytes), self._h)

    def launch_count(self) -> int:
        return int(load_library().dqgan_launch_count(self._h))

    def last_error(self) -> str:
        return load_library().dqgan_last_error(self._h).decode()


def create(cfg: Config) -> Handle:
    return Handle(cfg)


def topk_compress_noalloc(g, e, out_msg, d: int, k: int, lr: float, cuda_stream: int | None = None) -> None:
    """dqgan_topk_compress_noalloc: top-k worker step on a caller-owned residual,
    with no device allocation (scratch is a fixed array in the library)."""
    _check(load_library().dqgan_topk_compress_noalloc(_ptr(g), _ptr(e), _ptr(out_msg), d, k, lr,
                                                      cuda_stream))
