"""Benchmark of the DQGAN hot path (Algorithm 2: worker error-feedback +
compression of all M workers, then the fused server decode/average/update).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
                    [--impl reference] [--lookahead]

One step = dqgan_workers_compress_all over all M workers + dqgan_server_
aggregate_update, on fresh synthetic gradients already resident in HBM.
Gradient generation and an L2 flush (a 256 MB write) run between timed
regions and are not timed; each step's timed region is bracketed by CUDA
events on the stream the kernels run on.  The metric is updated parameters
per second, d * M per step, over all ranks.

Default workload: the d = 1e8, M = 32, sign-per-4096 stress configuration
(the largest that fits one GPU).  N > 1 (torchrun, one rank per GPU) runs N
independent replicas -- the simulated workers share nothing across GPUs --
and reports the whole-job rate over the max-over-ranks time.

--impl reference times the CPU oracle (the code as the tests use it) over
whole steps of the same workload on all host cores (worker steps and server
element ranges in parallel threads) and prints the same line with
"impl": "reference".
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2010_13359_gb300.workloads import SIGN, SQUANT, TOPK, IDENTITY, QSGD, WORKLOADS  # noqa: E402

METRIC = "updated params/sec (d*M per step) and achieved HBM GB/s vs GB300 roofline"
UNIT = "params/s"
FALLBACK_HBM_GBS = 6800.0
L2_BYTES = 129 << 20
COMPRESSOR_NAME = {SIGN: "sign", TOPK: "topk", SQUANT: "squant", IDENTITY: "identity", QSGD: "qsgd"}
KERNEL_SOURCE = {SIGN: "dense_compress.cu", SQUANT: "dense_compress.cu", IDENTITY: "dense_compress.cu",
                 TOPK: "topk.cu", QSGD: "dense_compress.cu"}


def parse_args():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--workload", default="stress_sign", choices=sorted(WORKLOADS))
    ap.add_argument("--impl", default="gpu", choices=["gpu", "reference"])
    ap.add_argument("--lookahead", action="store_true", help="also keep the lookahead offsets h")
    ap.add_argument("--no-e2e", action="store_true", help="skip the end-to-end (host buffers) phase")
    ap.add_argument("--e2e-mode", default="zerocopy", choices=["copy", "pipelined", "zerocopy"],
                    help="how host gradients reach the kernels: one bulk copy then compute; per-worker "
                         "copies on a second stream overlapped with per-worker compress; or the compress "
                         "kernels reading the pinned host buffer directly (NVLink-C2C)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--sweep", action="store_true",
                    help="instead of the one-line result, print one line per d = 2^16 .. 2^27 "
                         "(M = 8, sign per 1024, DCGAN gradient law): the roofline curve")
    ap.add_argument("--server", default="omd", choices=["omd", "oadam"],
                    help="server update: Algorithm 2's w = w - q_hat, or Optimistic Adam on q_hat "
                         "(alpha 1e-3, b1 0.5, b2 0.999, eps 1e-8, bias-corrected)")
    ap.add_argument("--override", action="append", default=[], metavar="FIELD=VALUE",
                    help="change a workload field (e.g. M=4 for a smaller profiling case)")
    return ap.parse_args()


def selected_workload(args):
    """The named workload, with integer fields changed by --override (for the
    smaller profiling cases); a changed d keeps the gradient distribution."""
    wl = WORKLOADS[args.workload]
    if not args.override:
        return wl
    kw = {}
    for item in args.override:
        key, val = item.split("=", 1)
        if key not in ("d", "M", "k", "bits", "bucket"):
            raise SystemExit(f"--override supports d, M, k, bits, bucket, not {key}")
        kw[key] = int(float(val))
    if "d" in kw and wl.segment_sizes is not None:
        kw.update(n_segments=1, segment_sizes=(kw["d"],), segment_std=wl.segment_std[:1])
    return wl.replace(name=wl.name + "[" + ",".join(args.override) + "]", **kw)


# ---------------------------------------------------------------------------
# bytes per step (algorithmic minimum)
# ---------------------------------------------------------------------------

def bucket_count(wl) -> int:
    if wl.layer_buckets:
        offs = wl.segment_offsets()
        return sum(-(-(b - a) // wl.bucket) for a, b in zip(offs[:-1], offs[1:]))
    return -(-wl.d // wl.bucket)


def message_payload_bytes(wl) -> int:
    nb = bucket_count(wl)
    if wl.compressor == SIGN:
        return 4 * nb + 4 * (-(-wl.d // 32))
    if wl.compressor in (SQUANT, QSGD):
        return 4 * nb + 4 * (-(-wl.d * wl.bits // 32))
    if wl.compressor == TOPK:
        return 8 * wl.k
    return 4 * wl.d


def compress_bytes(wl, lookahead: bool) -> int:
    """Per launch over all M workers: read g and e, write e (+h), write the message."""
    per_worker = 12 * wl.d + (4 * wl.d if lookahead else 0) + message_payload_bytes(wl)
    return wl.M * per_worker


OADAM = dict(alpha=1e-3, beta1=0.5, beta2=0.999, eps=1e-8)


def server_bytes(wl, oadam: bool = False) -> int:
    """Read and write w, read all M messages (top-k: read and write only the
    touched w); Optimistic Adam also reads and writes m, v, u_prev of every
    parameter (and so every w)."""
    if oadam:
        return 32 * wl.d + wl.M * message_payload_bytes(wl)
    if wl.compressor == TOPK:
        return wl.M * 8 * wl.k + 8 * min(wl.d, wl.M * wl.k)
    return 8 * wl.d + wl.M * message_payload_bytes(wl)


# ---------------------------------------------------------------------------
# environment helpers
# ---------------------------------------------------------------------------

def max_over_ranks(x: float, world: int, device=None) -> float:
    """The largest x over all ranks (all_reduce MAX; NCCL on GPUs, gloo on CPU)."""
    if world <= 1:
        return x
    import torch
    import torch.distributed as tdist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    tdist.all_reduce(t, op=tdist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(units_per_rank: int, steps: int, world: int, max_ms: float) -> float:
    """Units processed by all ranks per second, timed by the slowest rank."""
    return world * units_per_rank * steps / (max_ms / 1e3)


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def hbm_peak():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            v = float(json.load(f)["hbm_gbs"])
        return v, "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def source_digest(name: str) -> str:
    with open(os.path.join(ROOT, "paper_2010_13359_gb300", "csrc", name), "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()[:16]


def profiled_traffic(wl, kernel_file: str, units: int):
    """DRAM bytes per launch from the committed ncu summary of this workload,
    scaled to `units` parameters; None if absent or the kernel changed since."""
    path = os.path.join(ROOT, "profiles", f"ncu_compress_{wl.name}.md")
    if not os.path.exists(path):
        return None
    txt = open(path).read()
    m_b = re.search(r"dram_bytes_per_param\s*=\s*([0-9.eE+-]+)", txt)
    m_h = re.search(r"source_sha256_16\s*=\s*([0-9a-f]+)", txt)
    if not m_b or not m_h or m_h.group(1) != source_digest(kernel_file):
        return None
    return float(m_b.group(1)) * units


class ClockSampler:
    """nvidia-smi clocks / throttle reasons sampled every 200 ms while running."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.tmp = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=self.tmp, stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            time.sleep(0.25)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        self.tmp.flush()
        rows = []
        with open(self.tmp.name) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    rows.append((float(parts[1]), float(parts[2]), float(parts[3]), parts[4:9]))
                except ValueError:
                    continue
        os.unlink(self.tmp.name)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        loaded = [r for r in rows if r[2] > 200.0] or rows
        names = ["active_mask", "hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown",
                 "sw_power_cap"]
        reasons = set()
        for r in loaded:
            for name, val in zip(names[1:], r[3][1:]):
                if val.lower().startswith("active"):
                    reasons.add(name)
        return {"sm_mhz": statistics.median(r[0] for r in loaded), "sm_max_mhz": max(r[1] for r in rows),
                "reasons": sorted(reasons), "samples": len(loaded),
                "power_w_max": max(r[2] for r in rows)}


# ---------------------------------------------------------------------------
# CPU oracle timing (cpu_baseline leg and the reference arm)
# ---------------------------------------------------------------------------

def host_threads() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count() or 1


def cpu_model() -> str:
    """The host CPU's model name (lscpu, else /proc/cpuinfo, else the platform)."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.startswith("Model name:"):
                return line.split(":", 1)[1].strip()
    except Exception:
        pass
    try:
        with open("/proc/cpuinfo") as f:
            for line in f:
                if line.lower().startswith("model name"):
                    return line.split(":", 1)[1].strip()
    except Exception:
        pass
    import platform
    return platform.processor() or platform.machine()


class OracleSteps:
    """Whole steps of Algorithm 2 on the oracle, as the tests run it, spread
    over `threads` host threads: the M worker steps in parallel, then the
    server step in parallel element ranges (the oracle is a C library called
    through ctypes, which releases the GIL).  The gradients are one seeded
    batch generated up front (outside any timing) and used at every step."""

    def __init__(self, wl, threads: int, server: str = "omd"):
        from concurrent.futures import ThreadPoolExecutor

        import numpy as np

        import oracle

        self.np, self.oracle = np, oracle
        self.wl, self.threads = wl, threads
        segs = wl.segment_offsets() if wl.layer_buckets else None
        self.cfg = oracle.Config(d=wl.d, M=wl.M, compressor=wl.compressor, lr=wl.lr, bucket=wl.bucket,
                                 k=wl.k, bits=wl.bits, seed=wl.seed, segments=segs)
        self.pool = ThreadPoolExecutor(threads)
        self.E = np.zeros((wl.M, wl.d), np.float32)
        self.G = np.empty((wl.M, wl.d), np.float32)

        def gen(i):
            self.G[i] = wl.gradient_np(1, i)

        list(self.pool.map(gen, range(wl.M)))
        self.w = wl.w0_np()
        self.msgs = np.zeros((wl.M, oracle.message_bytes(self.cfg)), np.uint8)
        parts = 4 * threads
        cuts = sorted({wl.d * i // parts for i in range(parts + 1)})
        self.ranges = [(x, y) for x, y in zip(cuts[:-1], cuts[1:]) if y > x]
        self.opt = oracle.OAdamState(wl.d, oracle.OAdam(**OADAM)) if server == "oadam" else None
        self.t = 1

    def step(self) -> float:
        """One whole step; returns its wall time in seconds."""
        cfg, oracle, t = self.cfg, self.oracle, self.t

        def worker(i):
            self.msgs[i] = oracle.worker_step(cfg, i, t, self.G[i], self.E[i])

        t0 = time.perf_counter()
        list(self.pool.map(worker, range(self.wl.M)))
        if self.opt is None:
            list(self.pool.map(lambda r: oracle.server_step_range(cfg, self.msgs, self.w, r[0], r[1]), self.ranges))
        else:
            list(self.pool.map(lambda r: self.opt.server_step_range(cfg, t, self.msgs, self.w, r[0], r[1]),
                               self.ranges))
        dt = time.perf_counter() - t0
        self.t += 1
        return dt

    def close(self):
        self.pool.shutdown()
        self.E = self.G = self.msgs = None


def oracle_single_thread_estimate(wl, worker_fraction: float = 1 / 8, server_fraction: float = 1 / 64):
    """Single-thread oracle time for one full step of `wl`, estimated from a
    bounded sample: one worker step on a bucket-aligned prefix of the vector
    (`worker_fraction` of d; every worker's step costs the same per
    parameter) and the server step on a prefix (`server_fraction` of d),
    both scaled to all M workers and all of d."""
    import numpy as np

    import oracle

    def prefix(frac):
        if wl.compressor in (SIGN, SQUANT, QSGD):
            return min(wl.d, max(wl.bucket, int(wl.d * frac) // wl.bucket * wl.bucket))
        return min(wl.d, max(1, int(wl.d * frac)))

    def cfg_of(n):
        k = max(1, int(round(wl.k * n / wl.d))) if wl.compressor == TOPK else wl.k
        return oracle.Config(d=n, M=wl.M, compressor=wl.compressor, lr=wl.lr, bucket=wl.bucket, k=k,
                             bits=wl.bits, seed=wl.seed)

    rng = np.random.default_rng(1)
    wd = prefix(worker_fraction)
    g = (rng.standard_normal(wd, dtype=np.float32) * np.float32(1e-3)).astype(np.float32)
    e = np.zeros(wd, np.float32)
    t0 = time.perf_counter()
    oracle.worker_step(cfg_of(wd), 0, 1, g, e)
    t_worker = (time.perf_counter() - t0) * (wl.d / wd)
    sd = prefix(server_fraction)
    sub = cfg_of(sd)
    sub_msg = oracle.worker_step(sub, 0, 1, g[:sd].copy() if sd <= wd else
                                 rng.standard_normal(sd, dtype=np.float32), np.zeros(sd, np.float32))
    msgs = np.repeat(sub_msg[None, :], wl.M, axis=0)
    w = np.zeros(sd, np.float32)
    t0 = time.perf_counter()
    oracle.server_step(sub, msgs, w)
    t_server = (time.perf_counter() - t0) * (wl.d / sd)
    step = wl.M * t_worker + t_server
    sample = (f"projection, not a whole step: one worker step on {wd} of d = {wl.d} parameters "
              f"({t_worker:.2f} s scaled to d, x M = {wl.M}) + the server step on {sd} parameters "
              f"({t_server:.2f} s scaled to d); one host thread")
    return step, sample


def cpu_baseline_leg(wl, server: str = "omd"):
    """The GPU arm's cpu_baseline: one whole step of the workload on all host
    cores (timed after one untimed step), and the one-thread projection."""
    threads = host_threads()
    run = OracleSteps(wl, threads, server)
    run.step()
    dt = run.step()
    run.close()
    st1, sample1 = oracle_single_thread_estimate(wl)
    units = wl.d * wl.M
    return {"value": units / dt, "unit": UNIT, "cores": threads, "cpu_model": cpu_model(), "kind": "oracle",
            "sample": (f"one whole step of this workload (all M = {wl.M} worker steps and the server "
                       f"over all d = {wl.d}), timed after one untimed step, on {threads} host threads "
                       f"(worker steps and server element ranges in parallel): {dt:.2f} s"),
            "single_thread": {"value": units / st1, "unit": UNIT, "cores": 1, "sample": sample1}}


def run_reference(args, rank, world):
    """The oracle on the host cores, whole steps: W untimed, then K timed."""
    if rank != 0:
        return 0
    wl = selected_workload(args)
    threads = host_threads()
    run = OracleSteps(wl, threads, args.server)
    for _ in range(args.warmup):
        run.step()
    step_s = [run.step() for _ in range(args.steps)]
    run.close()
    total = sum(step_s)
    value = wl.d * wl.M * len(step_s) / total
    sample = (f"whole steps of this workload: {args.warmup} untimed, then {args.steps} timed, each all "
              f"M = {wl.M} worker steps and the server over all d = {wl.d}, on {threads} host threads "
              f"(worker steps and server element ranges in parallel); gradients: one seeded batch "
              f"generated before timing, used at every step")
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * total / len(step_s),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic", "config": workload_config(wl, args),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "cpu_model": cpu_model(),
                         "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def workload_config(wl, args):
    sets = max(1, min(args.steps + args.warmup, (4 << 30) // (wl.M * wl.d * 4)))
    big = compress_bytes(wl, args.lookahead) >= 2 * L2_BYTES
    c = {"workload": wl.name, "d": wl.d, "M": wl.M, "compressor": COMPRESSOR_NAME[wl.compressor],
         "lr": wl.lr, "gradients": f"{wl.dist}, {sets} seeded batch(es) generated before timing, used in turn",
         "lookahead": bool(args.lookahead),
         "l2": ("not flushed: every step reads and writes more than twice the 129 MB L2" if big else
                "flushed before every timed step (256 MB write, outside the timed region)"),
         "parallelism": f"replicas{args.gpus}" if args.gpus > 1 else "single",
         "server": ("optimistic_adam " + ", ".join(f"{k} {v:g}" for k, v in OADAM.items()) + ", bias-corrected"
                    if getattr(args, "server", "omd") == "oadam" else "omd: w = w - q_hat")}
    if wl.compressor in (SIGN, SQUANT, QSGD):
        c["bucket"] = wl.bucket
        c["buckets"] = "per layer segment" if wl.layer_buckets else "flat"
    if wl.compressor in (SQUANT, QSGD):
        c["bits"] = wl.bits
    if wl.compressor == TOPK:
        c["k"] = wl.k
    return c


# ---------------------------------------------------------------------------
# GPU arm
# ---------------------------------------------------------------------------

def run_gpu(args, rank, world, local):
    import torch
    import torch.distributed as tdist

    import paper_2010_13359_gb300 as P

    wl = selected_workload(args)
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        tdist.init_process_group("nccl", device_id=dev)

    def barrier():
        if world > 1:
            tdist.barrier()

    stream = torch.cuda.current_stream(dev)
    flags = P.KEEP_LOOKAHEAD if args.lookahead else 0
    h = P.create(P.make_config(d=wl.d, M=wl.M, compressor=wl.compressor, lr=wl.lr, bucket=wl.bucket,
                               k=wl.k, bits=wl.bits, seed=wl.seed, flags=flags,
                               cuda_stream=stream.cuda_stream))
    if wl.layer_buckets:
        h.set_segments(wl.segment_offsets())
    if args.server == "oadam":
        h.set_server_optimizer(P.dqgan.oadam(**OADAM))
    mb = h.message_bytes()
    msgs = torch.empty((wl.M, mb), dtype=torch.uint8, device=dev)
    w = wl.w0_torch(dev)
    std_vec = wl.std_vector_torch(dev) if wl.dist == "gauss" else None
    # Gradients: `sets` batches generated before any timing (up to 4 GB of
    # them), used in turn, so the timed loop only enqueues the two C-ABI calls
    # and the GPU never waits on the host.  A step that moves less than twice
    # the L2 size is preceded by a 256 MB L2 flush outside its timed region.
    sets = max(1, min(args.steps + args.warmup, (4 << 30) // (wl.M * wl.d * 4)))
    gs = [torch.empty((wl.M, wl.d), dtype=torch.float32, device=dev) for _ in range(sets)]
    for i, gi in enumerate(gs):
        wl.fill_gradients_torch(gi, i + 1, std_vec)
    g = gs[0]
    need_flush = compress_bytes(wl, args.lookahead) < 2 * L2_BYTES
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev) if need_flush else None

    def one_step(t, ev=None):
        gt = gs[(t - 1) % sets]
        if need_flush:
            flush.zero_()
        if ev:
            ev[0].record(stream)
        h.workers_compress_all(gt, wl.d, msgs)
        if ev:
            ev[1].record(stream)
        h.server_aggregate_update(msgs, w)
        if ev:
            ev[2].record(stream)

    for t in range(1, args.warmup + 1):
        one_step(t)
    torch.cuda.synchronize(dev)
    barrier()
    torch.cuda.synchronize(dev)
    events = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    with ClockSampler(local) as clk:
        launches0 = h.launch_count()
        if not need_flush:
            # The timed region: K steps back to back, events only at its ends
            # (an event between two kernels costs the second one its launch
            # overlap, 2-5 us, which small problems feel).
            ends[0].record(stream)
            for s in range(args.steps):
                one_step(args.warmup + 1 + s)
            ends[1].record(stream)
            torch.cuda.synchronize(dev)
        launches = h.launch_count() - launches0
        barrier()
        torch.cuda.synchronize(dev)
        launches1 = h.launch_count()
        if need_flush:
            # small problems: each step after an L2 flush, events around every launch
            for s in range(args.steps):
                one_step(args.warmup + 1 + s, events[s])
            torch.cuda.synchronize(dev)
            launches = h.launch_count() - launches1
        else:
            # per-kernel durations: K compress launches back to back, then K
            # server launches back to back, each run between two events
            kev = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
            kev[0].record(stream)
            for s in range(args.steps):
                h.workers_compress_all(gs[(args.warmup + s) % sets], wl.d, msgs)
            kev[1].record(stream)
            for s in range(args.steps):
                h.server_aggregate_update(msgs, w)
            kev[2].record(stream)
            torch.cuda.synchronize(dev)
    barrier()
    torch.cuda.synchronize(dev)
    if need_flush:
        comp_ms = [e[0].elapsed_time(e[1]) for e in events]
        serv_ms = [e[1].elapsed_time(e[2]) for e in events]
        region_ms = sum(c + s for c, s in zip(comp_ms, serv_ms))
    else:
        comp_ms = [kev[0].elapsed_time(kev[1]) / args.steps]
        serv_ms = [kev[1].elapsed_time(kev[2]) / args.steps]
        region_ms = ends[0].elapsed_time(ends[1])
    total_ms = max_over_ranks(region_ms, world, dev)
    units = wl.d * wl.M
    value = whole_job_rate(units, args.steps, world, total_ms)

    # end to end: host gradients (pinned) -> the C-ABI calls -> params -> host
    e2e = None
    if not args.no_e2e:
        g_host = torch.empty((wl.M, wl.d), dtype=torch.float32, pin_memory=True)
        w_host = torch.empty(wl.d, dtype=torch.float32, pin_memory=True)
        g_host.copy_(g)
        torch.cuda.synchronize(dev)
        e2e_steps = max(1, min(args.steps, 10))
        copy_stream = torch.cuda.Stream(dev)
        copied = [torch.cuda.Event() for _ in range(wl.M)]
        # the parameters go back on their own stream, overlapping the next
        # step's gradient reads (the link is full duplex); the next server
        # step waits for that copy before it updates w again
        back_stream = torch.cuda.Stream(dev)
        served, sent = torch.cuda.Event(), torch.cuda.Event()
        sent.record(back_stream)

        def e2e_step():
            if args.e2e_mode == "copy":
                g.copy_(g_host, non_blocking=True)
                h.workers_compress_all(g, wl.d, msgs)
            elif args.e2e_mode == "pipelined":
                copy_stream.wait_stream(stream)
                with torch.cuda.stream(copy_stream):
                    for i in range(wl.M):
                        g[i].copy_(g_host[i], non_blocking=True)
                        copied[i].record(copy_stream)
                for i in range(wl.M):
                    stream.wait_event(copied[i])
                    h.worker_compress(i, g[i], msgs[i])
            else:  # the kernels read the pinned host gradients in place
                h.workers_compress_all(g_host, wl.d, msgs)
            stream.wait_event(sent)
            h.server_aggregate_update(msgs, w)
            served.record(stream)
            back_stream.wait_event(served)
            with torch.cuda.stream(back_stream):
                w_host.copy_(w, non_blocking=True)
                sent.record(back_stream)

        e2e_step()
        torch.cuda.synchronize(dev)
        barrier()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(e2e_steps):
            e2e_step()
        stream.wait_event(sent)  # the last step's parameters are on the host
        b.record(stream)
        torch.cuda.synchronize(dev)
        e2e_ms = max_over_ranks(a.elapsed_time(b), world, dev)
        # the host link's own rate: a bulk copy of the same pinned gradients
        lk = min(g_host.numel(), 1 << 28)
        src, dst = g_host.view(-1)[:lk], g.view(-1)[:lk]
        dst.copy_(src, non_blocking=True)
        a.record(stream)
        for _ in range(3):
            dst.copy_(src, non_blocking=True)
        b.record(stream)
        torch.cuda.synchronize(dev)
        link_gbs = 3 * lk * 4 / (a.elapsed_time(b) * 1e6)
        h2d = int(g.numel() * 4)
        e2e = {"value": whole_job_rate(units, e2e_steps, world, e2e_ms), "unit": UNIT,
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": int(w.numel() * 4),
               "steps": e2e_steps, "ms_per_step": e2e_ms / e2e_steps, "mode": args.e2e_mode,
               "host_link": {"bound": "host-to-device link", "measured_gbs": link_gbs,
                             "achieved_gbs": h2d / (e2e_ms / e2e_steps * 1e6),
                             "frac": h2d / (e2e_ms / e2e_steps * 1e6) / link_gbs}}
        del g_host, w_host

    h.synchronize()
    h.destroy()
    if world > 1:
        tdist.destroy_process_group()
    if rank != 0:
        return 0

    peak, peak_kind = hbm_peak()
    comp_avg = statistics.mean(comp_ms)
    serv_avg = statistics.mean(serv_ms)
    cb = compress_bytes(wl, args.lookahead)
    sb = server_bytes(wl, args.server == "oadam")
    timing = ("CUDA events around each launch, each step after an L2 flush" if need_flush else
              f"CUDA events around {args.steps} launches of the kernel back to back, averaged")
    comp_gbs = cb / (comp_avg / 1e3) / 1e9
    serv_gbs = sb / (serv_avg / 1e3) / 1e9
    traffic = profiled_traffic(wl, KERNEL_SOURCE[wl.compressor], units) if not args.lookahead else None
    roofline = {"bound": "hbm", "kernel": f"{COMPRESSOR_NAME[wl.compressor]}_compress (all M workers)",
                "achieved": comp_gbs, "peak": peak, "unit": "GB/s", "frac": comp_gbs / peak,
                "traffic": traffic, "algorithmic_bytes": cb, "ms": comp_avg,
                "peak_source": f"{peak_kind} hbm_gbs", "timing": timing}
    roofline_server = {"bound": "hbm", "kernel": f"{COMPRESSOR_NAME[wl.compressor]}_server"
                                                  + ("_oadam" if args.server == "oadam" else ""),
                       "achieved": serv_gbs, "peak": peak, "unit": "GB/s", "frac": serv_gbs / peak,
                       "algorithmic_bytes": sb, "ms": serv_avg, "timing": timing}
    cpu = None
    if world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline_leg(wl, args.server)
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": total_ms / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": workload_config(wl, args), "roofline": roofline, "roofline_server": roofline_server,
        "cpu_baseline": cpu, "e2e": e2e, "gpu_launches": launches, "clocks": clk.summary(),
    }
    print(json.dumps(line), flush=True)
    return 0


def run_sweep(args):
    """Device-resident step time over d = 2^16 .. 2^27 (M = 8, sign per 1024)."""
    import torch

    import paper_2010_13359_gb300 as P
    from paper_2010_13359_gb300.workloads import sweep_workload

    dev = torch.device("cuda", 0)
    stream = torch.cuda.current_stream(dev)
    peak, peak_kind = hbm_peak()
    for log2_d in range(16, 28):
        wl = sweep_workload(log2_d)
        h = P.create(P.make_config(d=wl.d, M=wl.M, compressor=wl.compressor, lr=wl.lr, bucket=wl.bucket,
                                   seed=wl.seed, cuda_stream=stream.cuda_stream))
        g = torch.empty((wl.M, wl.d), dtype=torch.float32, device=dev)
        msgs = torch.empty((wl.M, h.message_bytes()), dtype=torch.uint8, device=dev)
        w = wl.w0_torch(dev)
        flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
        std_vec = wl.std_vector_torch(dev)
        comp, serv = [], []
        for t in range(1, args.warmup + args.steps + 1):
            wl.fill_gradients_torch(g, t, std_vec)
            flush.zero_()
            ev = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
            ev[0].record(stream)
            h.workers_compress_all(g, wl.d, msgs)
            ev[1].record(stream)
            h.server_aggregate_update(msgs, w)
            ev[2].record(stream)
            torch.cuda.synchronize(dev)
            if t > args.warmup:
                comp.append(ev[0].elapsed_time(ev[1]))
                serv.append(ev[1].elapsed_time(ev[2]))
        h.destroy()
        c_ms, s_ms = statistics.median(comp), statistics.median(serv)
        cb, sb = compress_bytes(wl, False), server_bytes(wl)
        print(json.dumps({"sweep": "sign_1024_M8", "d": wl.d, "M": wl.M, "params_per_s": wl.d * wl.M / ((c_ms + s_ms) / 1e3),
                          "compress_ms": c_ms, "compress_gbs": cb / c_ms / 1e6, "compress_frac": cb / c_ms / 1e6 / peak,
                          "server_ms": s_ms, "server_gbs": sb / s_ms / 1e6, "server_frac": sb / s_ms / 1e6 / peak,
                          "peak": peak, "peak_source": peak_kind}), flush=True)
    return 0


def main():
    args = parse_args()
    rank, world, local = dist_env()
    if args.impl == "reference":
        return run_reference(args, rank, world)
    if args.sweep:
        return run_sweep(args)
    return run_gpu(args, rank, world, local)


if __name__ == "__main__":
    sys.exit(main())
