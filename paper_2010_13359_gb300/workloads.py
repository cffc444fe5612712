"""Seeded synthetic inputs for the DQGAN hot path.

This module makes inputs only: flat gradient vectors shaped like the paper's
GAN workloads (a DCGAN-sized and a ResNet-GAN-sized generator+discriminator
parameter vector cut into layer segments with their own gradient scale), the
initial parameters, and the workload table.  It holds none of the method's
arithmetic and is shared by the CUDA-path tests, the oracle-side tests and
the benchmark, so that both sides see identical bytes.

The paper trains DCGAN on CIFAR-10 / CelebA (Section 4); neither the data
nor the models are available, so gradients are synthetic:

* the flat vector is cut into S contiguous "layer" segments whose sizes are
  drawn from the seed (weights 2^U(-3,3), normalised to d, multiples of 32,
  remainder to the last segment) unless the sizes are fixed;
* entries of segment l are N(0, std_l^2), std_l log-uniform in a range, or
  Student-t with nu = 3 (Z / sqrt(chi2_3 / 3)) times a scale for the
  heavy-tailed stress case;
* every (step, worker) pair has its own stream, keyed by the seed.
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np

SIGN, TOPK, SQUANT, IDENTITY, QSGD = 0, 1, 2, 3, 4


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    d: int
    M: int
    compressor: int
    bucket: int = 512
    k: int = 1
    bits: int = 8
    lr: float = 1e-3
    steps: int = 20
    seed: int = 20101335
    n_segments: int = 1
    segment_sizes: tuple | None = None     # fixed sizes, else drawn from the seed
    segment_std: tuple | None = None       # fixed stds, else log-uniform in std_range
    std_range: tuple = (1e-4, 1e-1)
    dist: str = "gauss"                    # "gauss" or "student_t3"
    dist_scale: float = 1.0
    w0_std: float = 0.02
    layer_buckets: bool = False            # buckets restart at every segment (per-layer bucketing)

    # -- layer segments ------------------------------------------------------
    def segments(self) -> tuple[list[int], list[float]]:
        rng = np.random.Generator(np.random.Philox(key=self.seed ^ 0x5E6))
        S = self.n_segments
        if self.segment_sizes is not None:
            sizes = list(self.segment_sizes)
        else:
            weights = 2.0 ** rng.uniform(-3.0, 3.0, size=S)
            raw = weights / weights.sum() * self.d
            sizes = [max(32, int(x) // 32 * 32) for x in raw[:-1]]
            sizes.append(self.d - sum(sizes))
            if sizes[-1] <= 0:
                raise ValueError("segment draw left no room for the last segment")
        if self.segment_std is not None:
            stds = list(self.segment_std)
        else:
            lo, hi = (math.log(x) for x in self.std_range)
            stds = [float(math.exp(v)) for v in rng.uniform(lo, hi, size=S)]
        assert sum(sizes) == self.d and len(sizes) == len(stds)
        return sizes, stds

    def segment_offsets(self) -> tuple:
        """0 = o_0 < o_1 < ... < o_S = d, the layer segment boundaries."""
        sizes, _ = self.segments()
        return tuple(int(x) for x in np.concatenate([[0], np.cumsum(sizes)]))

    def std_vector_np(self) -> np.ndarray:
        sizes, stds = self.segments()
        return np.repeat(np.asarray(stds, dtype=np.float32), sizes)

    def stream_seed(self, step: int, worker: int) -> int:
        return (self.seed * 1_000_003 + step * 7919 + worker * 104_729 + 1) & 0x7FFF_FFFF_FFFF

    # -- numpy generators (CPU-only tests) ------------------------------------
    def gradient_np(self, step: int, worker: int) -> np.ndarray:
        rng = np.random.Generator(np.random.Philox(key=self.stream_seed(step, worker)))
        if self.dist == "gauss":
            z = rng.standard_normal(self.d, dtype=np.float32)
            return (z * self.std_vector_np()).astype(np.float32)
        if self.dist == "student_t3":
            z = rng.standard_normal(self.d, dtype=np.float32)
            chi = sum(rng.standard_normal(self.d, dtype=np.float32) ** 2 for _ in range(3))
            return (z / np.sqrt(chi / np.float32(3.0)) * np.float32(self.dist_scale)).astype(np.float32)
        raise ValueError(self.dist)

    def gradients_np(self, step: int, workers=None) -> np.ndarray:
        ws = range(self.M) if workers is None else workers
        return np.stack([self.gradient_np(step, i) for i in ws])

    def w0_np(self) -> np.ndarray:
        rng = np.random.Generator(np.random.Philox(key=self.seed ^ 0xA11CE))
        return (rng.standard_normal(self.d, dtype=np.float32) * np.float32(self.w0_std)).astype(np.float32)

    # -- torch generators (device-resident inputs) ----------------------------
    def std_vector_torch(self, device):
        import torch
        sizes, stds = self.segments()
        return torch.repeat_interleave(torch.tensor(stds, dtype=torch.float32, device=device),
                                       torch.tensor(sizes, device=device))

    def fill_gradient_torch(self, out, step: int, worker: int, std_vec=None):
        """Write worker `worker`'s gradient of step `step` into the 1-D tensor `out`."""
        import torch
        gen = torch.Generator(device=out.device)
        gen.manual_seed(self.stream_seed(step, worker))
        if self.dist == "gauss":
            if std_vec is None:
                std_vec = self.std_vector_torch(out.device)
            torch.randn(out.shape, generator=gen, device=out.device, dtype=torch.float32, out=out)
            out.mul_(std_vec)
        elif self.dist == "student_t3":
            torch.randn(out.shape, generator=gen, device=out.device, dtype=torch.float32, out=out)
            chi = torch.zeros_like(out)
            tmp = torch.empty_like(out)
            for _ in range(3):
                torch.randn(out.shape, generator=gen, device=out.device, dtype=torch.float32, out=tmp)
                chi.addcmul_(tmp, tmp)
            chi.div_(3.0).sqrt_()
            out.div_(chi).mul_(self.dist_scale)
        else:
            raise ValueError(self.dist)
        return out

    def fill_gradients_torch(self, out, step: int, std_vec=None):
        """Fill an (M, >=d) tensor with every worker's gradient of step `step`."""
        if std_vec is None and self.dist == "gauss":
            std_vec = self.std_vector_torch(out.device)
        for i in range(self.M):
            self.fill_gradient_torch(out[i, : self.d], step, i, std_vec)
        return out

    def w0_torch(self, device):
        import torch
        gen = torch.Generator(device=device)
        gen.manual_seed(self.seed ^ 0xA11CE)
        return torch.randn(self.d, generator=gen, device=device, dtype=torch.float32) * self.w0_std

    def replace(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


def _dcgan(name, compressor, **kw):
    return Workload(name=name, d=3_600_000, M=8, compressor=compressor, steps=100,
                    n_segments=16, std_range=(1e-4, 1e-1), **kw)


def _resnet(name, bits, compressor=SQUANT):
    return Workload(name=name, d=25_000_000, M=16, compressor=compressor, bucket=512, bits=bits,
                    steps=50, n_segments=64, std_range=(1e-5, 1e-1))


WORKLOADS = {
    # d = 65,536 in 4 segments of 16,384 with fixed gradient stds; M = 4; sign per 512.
    "tiny_sign": Workload(name="tiny_sign", d=65_536, M=4, compressor=SIGN, bucket=512, steps=20,
                          n_segments=4, segment_sizes=(16_384,) * 4,
                          segment_std=(1e-1, 3e-2, 1e-2, 3e-3)),
    # DCGAN-scale generator+discriminator vector, d = 3.6M over 16 segments, M = 8.
    "dcgan_sign": _dcgan("dcgan_sign", SIGN, bucket=1024),
    "dcgan_topk": _dcgan("dcgan_topk", TOPK, k=36_000),
    # ResNet-GAN-scale vector, d = 25M over 64 segments, M = 16, b-bit quantiser per 512.
    "resnet_squant_b2": _resnet("resnet_squant_b2", 2),
    "resnet_squant_b4": _resnet("resnet_squant_b4", 4),
    "resnet_squant_b8": _resnet("resnet_squant_b8", 8),
    # Same vector with QSGD's l2-scaled quantiser (Eq. (qsgd)), 8 bits.
    "resnet_qsgd_b8": _resnet("resnet_qsgd_b8", 8, QSGD),
    # The same two vectors with buckets restarting at every layer segment.
    "dcgan_sign_layers": _dcgan("dcgan_sign_layers", SIGN, bucket=1024, layer_buckets=True),
    "resnet_squant_b8_layers": _resnet("resnet_squant_b8", 8).replace(name="resnet_squant_b8_layers",
                                                                       layer_buckets=True),
    # Heavy-tailed stress case: d = 1e8, M = 32, sign per 4096, Student-t(3) * 1e-3.
    "stress_sign": Workload(name="stress_sign", d=100_000_000, M=32, compressor=SIGN, bucket=4096,
                            steps=20, n_segments=1, segment_sizes=(100_000_000,),
                            segment_std=(1.0,), dist="student_t3", dist_scale=1e-3),
}


def game_diag_np(d: int, seed: int, lo: float = 0.5, hi: float = 1.5) -> np.ndarray:
    """The positive diagonal D (length d/2) of the bilinear game x^T D y."""
    rng = np.random.Generator(np.random.Philox(key=seed))
    return rng.uniform(lo, hi, size=d // 2).astype(np.float32)


def game_noise_np(d: int, seed: int, step: int, worker: int, std: float) -> np.ndarray:
    """The operator noise sigma * xi of worker `worker` at step `step`."""
    if std == 0.0:
        return np.zeros(d, np.float32)
    rng = np.random.Generator(np.random.Philox(key=(seed * 7919 + step * 131 + worker) & 0xFFFFFFFF))
    return (rng.standard_normal(d, dtype=np.float32) * np.float32(std)).astype(np.float32)


def sweep_workload(log2_d: int) -> Workload:
    """d = 2^log2_d, M = 8, sign per 1024, DCGAN gradient distribution."""
    return _dcgan(f"sweep_2^{log2_d}", SIGN, bucket=1024).replace(
        name=f"sweep_2^{log2_d}", d=2 ** log2_d, n_segments=16 if 2 ** log2_d >= 16 * 64 else 1)
