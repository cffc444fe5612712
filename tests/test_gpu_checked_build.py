"""The checked build (libdqgan_checked.so: the same sources compiled with
-DDQGAN_CHECK_BOUNDS).  Its kernels check the indices of the top-k path's
computed stores and loads -- candidate slots, message records, the server's
record offsets -- and skip an out-of-range access while setting a bit that
dqgan_synchronize reports as DQGAN_ERR_BOUNDS; its top-k scratch sits
between guard zones that dqgan_synchronize checks.  The guard-word tests and
the top-k parity tests run again in a child process with that library
loaded (the binding loads the library DQGAN_LIBRARY names) and must report
nothing; and a positive control -- a message whose last record lies past d,
which the normal build skips silently -- must come back as DQGAN_ERR_BOUNDS
with the context still usable."""
from __future__ import annotations

import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CONTROL = r"""
import numpy as np, torch
import paper_2010_13359_gb300 as P
assert P.dqgan.LIBRARY.endswith("libdqgan_checked.so"), P.dqgan.LIBRARY
dev = torch.device("cuda:0")
stream = torch.cuda.current_stream(dev)
d, M, k = 1000, 2, 4
h = P.create(P.make_config(d=d, M=M, compressor=P.TOPK, k=k, lr=0.1, cuda_stream=stream.cuda_stream))
mb = h.message_bytes()
rec = np.zeros((M, mb // 8, 2), np.uint32)
rec[0, :k, 0] = [1, 2, 3, d + 7]             # ascending; the last record lies past d
rec[1, :k, 0] = [10, 20, 30, 40]
rec[:, :k, 1] = np.float32(0.5).view(np.uint32)
msgs = torch.from_numpy(rec.view(np.uint8).reshape(M, mb)).to(dev)
w = torch.zeros(d, device=dev)
h.server_aggregate_update(msgs, w)
try:
    h.synchronize()
    raise SystemExit("the out-of-range record was not reported")
except P.DqganError as e:
    assert e.status == P.dqgan.ERR_BOUNDS, e
h.synchronize()                                # the word was cleared; the context is usable
assert float(w[1].item()) == -0.25 and float(w[10].item()) == -0.25
h.destroy()
print("control: DQGAN_ERR_BOUNDS")
"""


@pytest.fixture(scope="module")
def checked_env():
    from paper_2010_13359_gb300 import build
    path = build.build(checked=True)
    env = dict(os.environ, DQGAN_LIBRARY=path)
    return env


def test_checked_build_reports_an_out_of_range_record(checked_env):
    res = subprocess.run([sys.executable, "-c", CONTROL], cwd=ROOT, env=checked_env, capture_output=True,
                         text=True, timeout=600)
    assert res.returncode == 0, res.stdout + res.stderr
    assert "control: DQGAN_ERR_BOUNDS" in res.stdout


def test_guard_and_topk_tests_pass_under_the_checked_build(checked_env):
    cmd = [sys.executable, "-m", "pytest", "-q", "-x", "-m", "gpu", "-p", "no:cacheprovider",
           "tests/test_gpu_guards.py", "tests/test_gpu_topk_paths.py", "tests/test_gpu_parity.py", "-k",
           "guard or topk or Topk"]
    res = subprocess.run(cmd, cwd=ROOT, env=checked_env, capture_output=True, text=True, timeout=1500)
    assert res.returncode == 0, res.stdout[-4000:] + res.stderr[-2000:]
