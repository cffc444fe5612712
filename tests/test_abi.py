"""The C-ABI library on the host: it builds, loads without a GPU, exports every
symbol include/dqgan.h declares, its struct layout matches the header, and
its host-only calls (config validation, message layout) behave.  No call
here launches a kernel."""
from __future__ import annotations

import ctypes
import os
import re
import subprocess

import numpy as np
import pytest

import oracle

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "dqgan.h")


@pytest.fixture(scope="module")
def P():
    from paper_2010_13359_gb300 import build
    build.build()
    import paper_2010_13359_gb300 as P
    P.dqgan.load_library()
    return P


def declared_functions() -> list[str]:
    src = open(HEADER).read()
    return re.findall(r"DQGAN_API\s+[\w\s\*]+?\b(dqgan_\w+)\s*\(", src)


def test_header_declares_the_problem_statement_calls():
    names = declared_functions()
    for required in ["dqgan_create", "dqgan_worker_compress", "dqgan_server_aggregate_update",
                     "dqgan_destroy", "dqgan_workers_compress_all", "dqgan_worker_lookahead",
                     "dqgan_message_bytes", "dqgan_synchronize", "dqgan_get_residual",
                     "dqgan_set_residual", "dqgan_state_bytes", "dqgan_save_state", "dqgan_load_state",
                     "dqgan_last_error"]:
        assert required in names


def test_library_exports_every_declared_symbol(P):
    lib = ctypes.CDLL(P.dqgan.LIBRARY)
    for name in declared_functions():
        assert hasattr(lib, name), name
    out = subprocess.run(["nm", "-D", "--defined-only", P.dqgan.LIBRARY], capture_output=True, text=True)
    exported = set(re.findall(r" T (dqgan_\w+)", out.stdout))
    assert exported == set(declared_functions())


def test_config_struct_layout_matches_header(tmp_path, P):
    c = tmp_path / "layout.c"
    c.write_text("""
#include <stddef.h>
#include "dqgan.h"
_Static_assert(sizeof(dqgan_config) == 56, "size");
_Static_assert(offsetof(dqgan_config, d) == 0, "d");
_Static_assert(offsetof(dqgan_config, k) == 8, "k");
_Static_assert(offsetof(dqgan_config, lr) == 16, "lr");
_Static_assert(offsetof(dqgan_config, M) == 20, "M");
_Static_assert(offsetof(dqgan_config, compressor) == 24, "compressor");
_Static_assert(offsetof(dqgan_config, bucket) == 28, "bucket");
_Static_assert(offsetof(dqgan_config, bits) == 32, "bits");
_Static_assert(offsetof(dqgan_config, flags) == 36, "flags");
_Static_assert(offsetof(dqgan_config, seed) == 40, "seed");
_Static_assert(offsetof(dqgan_config, cuda_stream) == 48, "stream");
""")
    subprocess.run(["gcc", "-std=c11", "-fsyntax-only", "-I", os.path.join(ROOT, "include"), str(c)],
                   check=True)
    C = P.dqgan.Config
    for name, off in [("d", 0), ("k", 8), ("lr", 16), ("M", 20), ("compressor", 24), ("bucket", 28),
                      ("bits", 32), ("flags", 36), ("seed", 40), ("cuda_stream", 48)]:
        assert getattr(C, name).offset == off


@pytest.mark.parametrize("kw,needle", [
    (dict(d=0, M=1, compressor=0, bucket=512), "d ="),
    (dict(d=10, M=0, compressor=0, bucket=512), "M ="),
    (dict(d=10, M=5000, compressor=0, bucket=512), "M ="),
    (dict(d=10, M=1, compressor=0, bucket=100), "bucket"),
    (dict(d=10, M=1, compressor=0, bucket=16), "bucket"),
    (dict(d=10, M=1, compressor=0, bucket=8192), "bucket"),
    (dict(d=10, M=1, compressor=2, bucket=512, bits=3), "bits"),
    (dict(d=10, M=1, compressor=1, k=11), "k ="),
    (dict(d=10, M=1, compressor=1, k=0), "k ="),
    (dict(d=10, M=1, compressor=7), "compressor"),
    (dict(d=10, M=1, compressor=3, lr=float("nan")), "lr"),
    (dict(d=10, M=1, compressor=3, flags=2), "flag"),
])
def test_invalid_configs_are_rejected_on_the_host(P, kw, needle):
    cfg = P.make_config(**kw)
    with pytest.raises(P.DqganError) as ei:
        P.validate_config(cfg)
    assert ei.value.status == P.dqgan.ERR_INVALID_ARG
    assert needle in str(ei.value)
    # create refuses the same config before touching the GPU
    with pytest.raises(P.DqganError) as ei:
        P.create(cfg)
    assert ei.value.status == P.dqgan.ERR_INVALID_ARG


def test_message_layout_agrees_with_the_oracles_statement(P):
    rng = np.random.default_rng(0)
    for _ in range(300):
        comp = int(rng.integers(0, 4))
        d = int(rng.choice([1, 2, 31, 32, 33, 4095, 4097, 65537, 3_600_000, 25_000_000, 100_000_000]))
        bucket = int(2 ** rng.integers(5, 13))
        bits = int(rng.choice([2, 4, 8]))
        k = int(rng.integers(1, d + 1))
        cfg = P.make_config(d=d, M=3, compressor=comp, bucket=bucket, bits=bits, k=k)
        got = P.message_layout(cfg)
        want = oracle.layout(oracle.Config(d=d, M=3, compressor=comp, bucket=bucket, bits=bits, k=k))
        assert got == want
        assert got[2] % 256 == 0 and got[1] % 256 == 0


def test_missing_library_fails_loudly(P, tmp_path):
    import importlib
    mod = importlib.import_module("paper_2010_13359_gb300.dqgan")
    saved = mod._lib
    mod._lib = None
    try:
        with pytest.raises(RuntimeError, match="missing"):
            mod.load_library(str(tmp_path / "libdqgan.so"))
    finally:
        mod._lib = saved


def test_server_optimizer_struct_layout_matches_header(tmp_path, P):
    c = tmp_path / "opt.c"
    c.write_text("""
#include <stddef.h>
#include "dqgan.h"
_Static_assert(sizeof(dqgan_server_optimizer) == 28, "size");
_Static_assert(offsetof(dqgan_server_optimizer, kind) == 0, "kind");
_Static_assert(offsetof(dqgan_server_optimizer, flags) == 4, "flags");
_Static_assert(offsetof(dqgan_server_optimizer, alpha) == 8, "alpha");
_Static_assert(offsetof(dqgan_server_optimizer, beta1) == 12, "beta1");
_Static_assert(offsetof(dqgan_server_optimizer, beta2) == 16, "beta2");
_Static_assert(offsetof(dqgan_server_optimizer, eps) == 20, "eps");
_Static_assert(DQGAN_SERVER_OMD == 0 && DQGAN_SERVER_OADAM == 1, "kinds");
_Static_assert(DQGAN_OADAM_ADAPTIVE == 1u && DQGAN_OADAM_BIAS_CORRECTION == 2u, "flags");
""")
    subprocess.run(["gcc", "-std=c11", "-fsyntax-only", "-I", os.path.join(ROOT, "include"), str(c)],
                   check=True)
    S = P.dqgan.ServerOptimizer
    for name, off in [("kind", 0), ("flags", 4), ("alpha", 8), ("beta1", 12), ("beta2", 16), ("eps", 20)]:
        assert getattr(S, name).offset == off


def test_server_optimizer_calls_reject_a_null_handle(P):
    L = P.dqgan.load_library()
    opt = P.dqgan.oadam(1e-3, 0.5, 0.999, 1e-8)
    import ctypes
    assert L.dqgan_set_server_optimizer(None, ctypes.byref(opt)) == P.dqgan.ERR_INVALID_ARG
    assert L.dqgan_get_server_state(None, 0, None) == P.dqgan.ERR_INVALID_ARG
    assert b"NULL" in L.dqgan_last_error(None)


def test_sharding_calls_reject_a_null_handle(P):
    L = P.dqgan.load_library()
    assert L.dqgan_set_local_workers(None, 0, 1) == P.dqgan.ERR_INVALID_ARG
    assert L.dqgan_workers_compress_range(None, 0, 1, None, 4, None) == P.dqgan.ERR_INVALID_ARG
    assert b"NULL" in L.dqgan_last_error(None)


def test_status_codes_match_the_header(P):
    hdr = open(os.path.join(ROOT, "include", "dqgan.h")).read()
    for name in ("OK", "ERR_INVALID_ARG", "ERR_OOM", "ERR_CUDA", "ERR_UNSUPPORTED", "ERR_TIMEOUT", "ERR_BOUNDS"):
        m = re.search(r"#define DQGAN_%s \(?(-?\d+)\)?" % name, hdr)
        assert m, name
        assert int(m.group(1)) == getattr(P.dqgan, name), name
