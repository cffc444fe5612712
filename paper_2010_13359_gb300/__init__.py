"""GB300-native (sm_103a) hot path of DQGAN (arXiv 2010.13359, Algorithm 2).

The compute lives in ``libdqgan.so`` (CUDA kernels behind the C-ABI of
``include/dqgan.h``); ``dqgan`` is its ctypes binding and ``workloads`` makes
the seeded synthetic inputs; ``games`` closes Algorithm 2 around a min-max
operator (the bilinear game of Section 2.2).
"""
from . import dqgan  # noqa: F401
from .dqgan import (  # noqa: F401
    ERR_TIMEOUT, IDENTITY, KEEP_LOOKAHEAD, QSGD, SIGN, SQUANT, TOPK, Config, DqganError, Handle, create, make_config,
    message_layout, validate_config,
)
