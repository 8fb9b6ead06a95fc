"""Seeded synthetic inputs shared by the CUDA path, the oracle, the tests and the bench.

This module holds none of the method's arithmetic: it only draws the data the
method runs on, from numpy's PCG64 generator with a stated seed.  The data
stand in for the paper's image-classification workloads (CIFAR-10 / ImageNet
CNN training, Sec. IV), which are not available: every replica holds a flat
fp32 parameter vector sized like a CNN, and the objective is the separable
quadratic f(x) = 1/2 sum_j h_j (x_j - c_j)^2, whose curvatures h_j and minimiser
c_j are drawn here.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

DEFAULT_SEED = 0x2007061340000001


@dataclass(frozen=True)
class Workload:
    """One synthetic workload: sizes, objective distributions and SGD knobs."""
    name: str
    n: int                 # replicas (the paper's nodes)
    P: int                 # parameters per replica
    K: int                 # iterations
    h_dist: str            # "uniform:a:b" or "loguniform:a:b"
    c_sigma: float         # c_j ~ N(0, c_sigma^2)
    sigma: float           # gradient-noise scale
    mu: float              # momentum
    wd: float              # weight decay
    lr0: float             # initial step size
    milestones: tuple = () # iterations where the step size is multiplied by lr_factor
    lr_factor: float = 0.1
    p_init: int = 4        # Algorithm 2's p_init (Sec. IV-B uses 4)
    K_s_frac: float = 0.25 # K_s = K_s_frac * K (Sec. IV-B uses 0.25K)
    cpsgd_p: int = 8       # the comparison constant period
    noise: str = "philox"  # "philox" (fresh per step) or "bf16" (pre-materialised tensor)
    seed: int = DEFAULT_SEED
    extra: dict = field(default_factory=dict)

    @property
    def K_s(self) -> int:
        return int(round(self.K_s_frac * self.K))


# The five synthetic workloads (n replicas of a CNN-sized fp32 vector).
WORKLOADS = {
    # n=4, P=2^20, h~U[0.1,1], c~N(0,1), noise N(0,0.5^2), momentum 0.9, lr 0.05, 100 iterations.
    "quadratic-n4-P1M": Workload("quadratic-n4-P1M", 4, 1 << 20, 100, "uniform:0.1:1", 1.0, 0.5,
                                 0.9, 0.0, 0.05, cpsgd_p=4),
    # n=8, ResNet-18-sized P, h~U[0.01,1], noise sigma 1, wd 5e-4, lr 0.1 x0.1 at 50% / 75% of 2000.
    "resnet18-n8": Workload("resnet18-n8", 8, 11_689_512, 2000, "uniform:0.01:1", 1.0, 1.0, 0.9,
                            5e-4, 0.1, milestones=(1000, 1500)),
    # n=16, ResNet-50-sized P, pre-materialised bf16 N(0,1) noise, lr 0.05, 1000 iterations.
    "resnet50-n16-bf16noise": Workload("resnet50-n16-bf16noise", 16, 25_557_032, 1000,
                                       "uniform:0.1:1", 1.0, 1.0, 0.9, 0.0, 0.05, noise="bf16"),
    # n=8, VGG-16-sized P, h~LogUniform[1e-3,1], c~N(0,0.1^2), sigma 0.5, wd 5e-4, 500 iterations.
    "vgg16-n8": Workload("vgg16-n8", 8, 138_357_544, 500, "loguniform:0.001:1", 0.1, 0.5, 0.9,
                         5e-4, 0.05),
}

# The schedule study of Sec. III: 16 replicas, 4000 iterations, step size 0.1 x0.1 at 50 % and 75 %
# of the run (the GoogLeNet / CIFAR-10 schedule of Sec. III-A on a 2^20-parameter surrogate).
WORKLOADS["strategies-n16"] = Workload("strategies-n16", 16, 1 << 20, 4000, "uniform:0.01:1", 1.0, 1.0, 0.9,
                                       5e-4, 0.1, milestones=(2000, 3000), K_s_frac=0.25)

SWEEP_N = (2, 4, 8, 16, 32)
SWEEP_LOG2P = (16, 18, 20, 22, 24, 26, 28)


def _rng(seed: int, stream: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64([seed & 0xFFFFFFFFFFFFFFFF, stream]))


def draw_h(P: int, dist: str, seed: int) -> np.ndarray:
    """Curvatures h_j (fp32) from "uniform:a:b" or "loguniform:a:b"."""
    kind, a, b = dist.split(":")
    a, b = float(a), float(b)
    u = _rng(seed, 1).random(P, dtype=np.float32)
    if kind == "uniform":
        return (np.float32(a) + np.float32(b - a) * u).astype(np.float32)
    if kind == "loguniform":
        la, lb = np.log(a), np.log(b)
        return np.exp(la + (lb - la) * u.astype(np.float64)).astype(np.float32)
    raise ValueError(dist)


def draw_c(P: int, c_sigma: float, seed: int) -> np.ndarray:
    """Minimisers c_j ~ N(0, c_sigma^2) (fp32)."""
    z = _rng(seed, 2).standard_normal(P, dtype=np.float32)
    return (np.float32(c_sigma) * z).astype(np.float32)


def problem(w: Workload, P: int | None = None):
    """(h, c) for a workload; P overrides the size for scaled-down cases."""
    P = w.P if P is None else P
    return draw_h(P, w.h_dist, w.seed), draw_c(P, w.c_sigma, w.seed)


def zero_state(n: int, P: int):
    """x_0 = 0 shared by every replica, v_0 = 0."""
    return np.zeros((n, P), np.float32), np.zeros((n, P), np.float32)


def random_state(n: int, P: int, seed: int, scale: float = 1.0, spread: float = 0.1):
    """A mid-run state: replicas near a common point, momentum buffers nonzero."""
    r = _rng(seed, 3)
    base = r.standard_normal(P, dtype=np.float32) * np.float32(scale)
    x = (base[None, :] + np.float32(spread) * r.standard_normal((n, P), dtype=np.float32))
    v = np.float32(0.1) * r.standard_normal((n, P), dtype=np.float32)
    return np.ascontiguousarray(x, np.float32), np.ascontiguousarray(v, np.float32)


def sweep_replicas(n: int, P: int, seed: int, offset: float = 1e-3, shared: bool = False):
    """Replicas x_i = N(0,1) + i * offset: independent draws per replica, or one shared draw."""
    r = _rng(seed, 4)
    if shared:
        base = r.standard_normal(P, dtype=np.float32)
        x = np.empty((n, P), np.float32)
        for i in range(n):
            x[i] = base + np.float32(i * offset)
        return x
    x = r.standard_normal((n, P), dtype=np.float32)
    for i in range(n):
        x[i] += np.float32(i * offset)
    return x
