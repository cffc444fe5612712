"""CUDA path vs oracle on the paper-shaped workloads at their full sizes, over
whole runs, in the launch configuration the benchmark times
(dqgan_workers_compress_all over all M workers, then
dqgan_server_aggregate_update).

Every workload runs free on both sides for its whole run (Algorithm 2,
Section 3.1): the GPU generates each step's gradients, the oracle gets the
same bytes, and at every step every worker's message is compared bit for
bit and the parameters w are compared against the stated tolerance (max
relative error 1e-5 per element per step, 1e-4 after the run) and then bit
for bit -- both sides take the server's sum in the same fixed order.  At the
end every worker's residual e is compared bit for bit.

* tiny sign (d = 65,536, M = 4, 20 steps), DCGAN-scale sign (d = 3.6M,
  M = 8, 100 steps), top-k (k = 36,000, 100 steps), and the same sign
  vector with per-layer buckets;
* ResNet-GAN-scale stochastic quantiser (d = 25M, M = 16, b = 2, 4, 8, 50
  steps), QSGD's l2 scale at b = 8, and b = 8 with per-layer buckets;
* the stress case (d = 1e8, M = 32, Student-t gradients, 20 steps);
* the d sweep's sizes (2^16, 2^21, 2^27 at M = 8), a few steps each.

The oracle's worker steps and server element ranges run on a thread pool
(the oracle is a C library called through ctypes, which releases the GIL).
"""
from __future__ import annotations

import os
from concurrent.futures import ThreadPoolExecutor

import numpy as np
import pytest

import oracle
from parity_helpers import RUN_RTOL, STEP_RTOL, assert_bits_equal, assert_messages_equal, assert_params_equal
from paper_2010_13359_gb300.workloads import WORKLOADS, sweep_workload

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

THREADS = max(1, min(16, os.cpu_count() or 1))


@pytest.fixture(scope="module")
def P():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2010_13359_gb300 as P
    return P


@pytest.fixture(scope="module")
def pool():
    with ThreadPoolExecutor(THREADS) as ex:
        yield ex


def ocfg_of(wl):
    segs = wl.segment_offsets() if wl.layer_buckets else None
    return oracle.Config(d=wl.d, M=wl.M, compressor=wl.compressor, lr=wl.lr, bucket=wl.bucket, k=wl.k,
                         bits=wl.bits, seed=wl.seed, segments=segs)


def handle_of(P, wl, stream):
    h = P.create(P.make_config(d=wl.d, M=wl.M, compressor=wl.compressor, lr=wl.lr, bucket=wl.bucket,
                               k=wl.k, bits=wl.bits, seed=wl.seed, cuda_stream=stream.cuda_stream))
    if wl.layer_buckets:
        h.set_segments(wl.segment_offsets())
    return h


def oracle_server(pool, ocfg, msgs, w):
    """Oracle server step of Algorithm 2 on w in place, element ranges on the pool."""
    parts = 4 * THREADS
    cuts = sorted({ocfg.d * i // parts for i in range(parts + 1)})
    ranges = [(a, b) for a, b in zip(cuts[:-1], cuts[1:]) if b > a]
    list(pool.map(lambda ab: oracle.server_step_range(ocfg, msgs, w, ab[0], ab[1]), ranges))


def whole_run(P, pool, wl, steps):
    ocfg = ocfg_of(wl)
    dev = torch.device("cuda:0")
    stream = torch.cuda.current_stream(dev)
    h = handle_of(P, wl, stream)
    mb = h.message_bytes()
    assert mb == oracle.message_bytes(ocfg)
    M, d = wl.M, wl.d
    w_gpu = wl.w0_torch(dev)
    w_orc = w_gpu.cpu().numpy().copy()
    g_dev = torch.empty((M, d), dtype=torch.float32, device=dev)
    msgs = torch.empty((M, mb), dtype=torch.uint8, device=dev)
    g_host = torch.empty((M, d), dtype=torch.float32, pin_memory=True)
    G = g_host.numpy()
    E = np.zeros((M, d), np.float32)
    std_vec = wl.std_vector_torch(dev) if wl.dist == "gauss" else None
    for t in range(1, steps + 1):
        wl.fill_gradients_torch(g_dev, t, std_vec)
        h.workers_compress_all(g_dev, d, msgs)
        h.server_aggregate_update(msgs, w_gpu)
        g_host.copy_(g_dev)
        got = msgs.cpu().numpy()

        def worker(i):
            want = oracle.worker_step(ocfg, i, t, G[i], E[i])
            assert_messages_equal(ocfg, got[i], want, f"{wl.name} worker {i} step {t}")
            return want

        want_msgs = np.stack(list(pool.map(worker, range(M))))
        oracle_server(pool, ocfg, want_msgs, w_orc)
        assert_params_equal(w_gpu.cpu().numpy(), w_orc, f"{wl.name} step {t}", STEP_RTOL)
    assert_params_equal(w_gpu.cpu().numpy(), w_orc, f"{wl.name} after {steps} steps", RUN_RTOL)
    e_i = np.empty(d, np.float32)
    for i in range(M):
        h.get_residual(i, e_i)
        assert_bits_equal(e_i, E[i], f"{wl.name} final residual worker {i}")
    h.destroy()


@pytest.mark.parametrize("name,steps", [
    ("tiny_sign", 20),
    ("dcgan_sign", 100),
    ("dcgan_sign_layers", 100),
    ("dcgan_topk", 100),
    ("resnet_squant_b2", 50),
    ("resnet_squant_b4", 50),
    ("resnet_squant_b8", 50),
    ("resnet_qsgd_b8", 50),
    ("resnet_squant_b8_layers", 50),
    ("stress_sign", 20),
])
def test_whole_run(P, pool, name, steps):
    whole_run(P, pool, WORKLOADS[name], steps)


@pytest.mark.parametrize("log2_d,steps", [(16, 5), (21, 5), (27, 3)])
def test_sweep_sizes(P, pool, log2_d, steps):
    whole_run(P, pool, sweep_workload(log2_d), steps)
