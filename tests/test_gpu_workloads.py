"""CUDA path vs oracle on the paper-shaped workloads at their full sizes, in
the launch configuration the benchmark times (dqgan_workers_compress_all over
all M workers, then dqgan_server_aggregate_update).

* tiny sign (d = 65,536, M = 4, 20 steps) and DCGAN-scale sign (d = 3.6M,
  M = 8, 100 steps) run free for the whole run on both sides: every message
  of every worker at every step bit for bit, final residuals bit for bit,
  parameters within 1e-5 per step and 1e-4 at the end;
* DCGAN-scale top-k (k = 36,000) the same over its first 20 steps;
* ResNet-GAN-scale stochastic quantiser (d = 25M, M = 16, b = 2, 4, 8) and
  the stress case (d = 1e8, M = 32, Student-t gradients): sampled workers
  run free for the first steps, then step-locked checks (oracle started from
  the GPU's own residual) at the last step, and the server step is checked
  on bucket-aligned slices of the parameter vector.
"""
from __future__ import annotations

import multiprocessing as mp

import numpy as np
import pytest

import oracle
from oracle_pool import worker_trajectory
from parity_helpers import (RUN_RTOL, STEP_RTOL, assert_bits_equal, assert_messages_equal, rel_err,
                            slice_messages)
from paper_2010_13359_gb300.workloads import WORKLOADS

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def P():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2010_13359_gb300 as P
    return P


def ocfg_of(wl):
    return oracle.Config(d=wl.d, M=wl.M, compressor=wl.compressor, lr=wl.lr, bucket=wl.bucket, k=wl.k,
                         bits=wl.bits, seed=wl.seed)


def handle_of(P, wl, stream):
    return P.create(P.make_config(d=wl.d, M=wl.M, compressor=wl.compressor, lr=wl.lr, bucket=wl.bucket,
                                  k=wl.k, bits=wl.bits, seed=wl.seed, cuda_stream=stream.cuda_stream))


@pytest.mark.parametrize("name,steps", [("tiny_sign", 20), ("dcgan_sign", 100), ("dcgan_topk", 20)])
def test_free_running_whole_run(P, name, steps):
    wl = WORKLOADS[name]
    ocfg = ocfg_of(wl)
    ctx = mp.get_context("spawn")
    with ctx.Pool(min(wl.M, 16)) as pool:
        traj = pool.map(worker_trajectory, [(name, {}, i, steps) for i in range(wl.M)])
    dev = torch.device("cuda:0")
    stream = torch.cuda.current_stream(dev)
    h = handle_of(P, wl, stream)
    mb = h.message_bytes()
    w0 = wl.w0_np()
    w_gpu = torch.from_numpy(w0.copy()).to(dev)
    w_orc = w0.copy()
    g_dev = torch.empty((wl.M, wl.d), dtype=torch.float32, device=dev)
    msgs = torch.empty((wl.M, mb), dtype=torch.uint8, device=dev)
    for t in range(1, steps + 1):
        g_dev.copy_(torch.from_numpy(wl.gradients_np(t)))
        h.workers_compress_all(g_dev, wl.d, msgs)
        h.server_aggregate_update(msgs, w_gpu)
        got = msgs.cpu().numpy()
        step_msgs = np.stack([traj[i][0][t - 1] for i in range(wl.M)])
        for i in range(wl.M):
            assert_messages_equal(ocfg, got[i], step_msgs[i], f"{name} worker {i} step {t}")
        oracle.server_step(ocfg, step_msgs, w_orc)
        err = rel_err(w_gpu.cpu().numpy(), w_orc)
        assert err <= STEP_RTOL, f"{name} step {t}: params rel err {err}"
    for i in range(wl.M):
        e_i = np.empty(wl.d, np.float32)
        h.get_residual(i, e_i)
        assert_bits_equal(e_i, traj[i][1], f"{name} final residual worker {i}")
    assert rel_err(w_gpu.cpu().numpy(), w_orc) <= RUN_RTOL
    h.destroy()


def sampled_run(P, wl, steps, free_steps, sample, slices, locked_steps):
    """Runs `steps` GPU steps on GPU-generated gradients; sampled workers run
    free on the oracle for `free_steps`; at `locked_steps` the sampled
    workers are re-checked from the GPU's own residual and the server step
    is checked on the given element slices."""
    ocfg = ocfg_of(wl)
    dev = torch.device("cuda:0")
    stream = torch.cuda.current_stream(dev)
    h = handle_of(P, wl, stream)
    mb = h.message_bytes()
    w_gpu = wl.w0_torch(dev)
    g_dev = torch.empty((wl.M, wl.d), dtype=torch.float32, device=dev)
    msgs = torch.empty((wl.M, mb), dtype=torch.uint8, device=dev)
    std_vec = wl.std_vector_torch(dev) if wl.dist == "gauss" else None
    e_free = {i: np.zeros(wl.d, np.float32) for i in sample}
    for t in range(1, steps + 1):
        wl.fill_gradients_torch(g_dev, t, std_vec)
        locked = t in locked_steps
        e_before = {}
        if locked:
            for i in sample:
                e_before[i] = np.empty(wl.d, np.float32)
                h.get_residual(i, e_before[i])
        h.workers_compress_all(g_dev, wl.d, msgs)
        w_before = w_gpu.cpu().numpy() if locked or t <= free_steps else None
        h.server_aggregate_update(msgs, w_gpu)
        if t <= free_steps or locked:
            got = msgs.cpu().numpy()
            for i in sample:
                g_i = g_dev[i].cpu().numpy()
                if t <= free_steps:
                    want = oracle.worker_step(ocfg, i, t, g_i, e_free[i])
                    assert_messages_equal(ocfg, got[i], want, f"{wl.name} free worker {i} step {t}")
                    e_gpu = np.empty(wl.d, np.float32)
                    h.get_residual(i, e_gpu)
                    assert_bits_equal(e_gpu, e_free[i], f"{wl.name} free residual {i} step {t}")
                if locked:
                    e_i = e_before[i]
                    want = oracle.worker_step(ocfg, i, t, g_i, e_i)
                    assert_messages_equal(ocfg, got[i], want, f"{wl.name} locked worker {i} step {t}")
                    e_gpu = np.empty(wl.d, np.float32)
                    h.get_residual(i, e_gpu)
                    assert_bits_equal(e_gpu, e_i, f"{wl.name} locked residual {i} step {t}")
            w_after = w_gpu.cpu().numpy()
            for a, b in slices:
                sub, sub_msgs = slice_messages(ocfg, got, a, b)
                w_ref = w_before[a:b].copy()
                oracle.server_step(sub, sub_msgs, w_ref)
                err = rel_err(w_after[a:b], w_ref)
                assert err <= STEP_RTOL, f"{wl.name} server step {t} slice [{a},{b}): {err}"
    h.destroy()


@pytest.mark.parametrize("bits", [2, 4, 8])
def test_resnet_squant_sampled(P, bits):
    wl = WORKLOADS[f"resnet_squant_b{bits}"]
    d = wl.d
    slices = [(0, 512 * 4096), (d // 2 // 512 * 512, d // 2 // 512 * 512 + 512 * 2048),
              ((d - 1_000_000) // 512 * 512, d)]
    sampled_run(P, wl, steps=wl.steps, free_steps=2, sample=[0, wl.M - 1], slices=slices,
                locked_steps={wl.steps})


def test_resnet_qsgd_sampled(P):
    wl = WORKLOADS["resnet_qsgd_b8"]
    d = wl.d
    slices = [(0, 512 * 4096), ((d - 1_000_000) // 512 * 512, d)]
    sampled_run(P, wl, steps=10, free_steps=2, sample=[0, wl.M - 1], slices=slices, locked_steps={10})


def test_stress_sign_sampled(P):
    wl = WORKLOADS["stress_sign"]
    d = wl.d
    slices = [(0, 4096 * 1024), (d // 2 // 4096 * 4096, d // 2 // 4096 * 4096 + 4096 * 512),
              ((d - 3_000_000) // 4096 * 4096, d)]
    sampled_run(P, wl, steps=wl.steps, free_steps=2, sample=[0, 1, wl.M - 1], slices=slices,
                locked_steps={1, wl.steps})


def test_dcgan_topk_locked_at_last_step(P):
    wl = WORKLOADS["dcgan_topk"]
    sampled_run(P, wl, steps=wl.steps, free_steps=0, sample=[0, wl.M - 1], slices=[],
                locked_steps={wl.steps // 2, wl.steps})
