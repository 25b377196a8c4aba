"""Seeded synthetic workloads for the GMC / GMC+ step.

This module only draws inputs: the initial parameters w_0 and the per-step
stochastic gradients g_{t,k} that Algorithm 1 (and Algorithm 2) take from the
workers' mini-batches. It holds none of the method's arithmetic, so both the
oracle side and the CUDA side may use it.

The paper trains ResNet20 / ViT on CIFAR (Sec. 5); no dataset is available here,
so gradients are synthetic and shaped like those models' gradients: the
parameter vector is cut into layer segments, each with its own gradient scale
(log-uniform), optionally with heavy-tailed noise and a per-worker non-IID mean
offset that stands in for the paper's Dirichlet non-IID split.

Two generators produce the same distributions from different random streams:
  * ``numpy``: host arrays, used where the oracle needs the very same inputs
    (all parity tests that run the oracle on a whole trajectory);
  * ``torch``: device tensors, used for the timed runs, where drawing
    gigabytes on the host would dominate the run time.
Within one generator every value is a pure function of (seed, workload, t).
"""
from __future__ import annotations

import dataclasses
import math
from typing import Optional

import numpy as np

__all__ = ["Workload", "WORKLOADS", "workload", "segment_sizes", "element_scale",
           "init_params", "NumpyGradients", "TorchGradients"]


@dataclasses.dataclass(frozen=True)
class Workload:
    """One benchmark configuration of a GMC / GMC+ step."""
    name: str
    d: int                      # parameters
    K: int                      # simulated workers
    compressor: str             # "topk", "topk_approx" or "rbgs"
    ratio: float                # top-k: k = max(1, floor(ratio*d)); rbgs: share of blocks
    beta: float
    eta: float
    steps: int
    block: int = 4096           # RBGS block size B
    lam: float = 0.0            # GMC+ detach coefficient (0 = GMC)
    per_worker: bool = False    # RBGS: per-worker block choice instead of a shared seed
    n_segments: int = 1         # layer segments (1 and iid=True: plain N(0,1))
    scale_lo: float = 1e-3      # per-segment gradient std ~ log-uniform [scale_lo, scale_hi]
    scale_hi: float = 1e-1
    big_segment: int = 0        # size of one forced segment (0 = none)
    laplace_frac: float = 0.0   # share of heavy-tailed (Laplace) noise draws
    laplace_scale: float = 5.0  # Laplace scale as a multiple of the segment std
    noniid: float = 0.0         # per-worker mean offset std as a multiple of the segment std
    iid_unit: bool = False      # gradients N(0,1) i.i.d., no segments
    w0_std: float = 0.01
    grad_dtype: str = "f32"     # gradient input: "f32", or "bf16" (gmc_step_bf16: half the bytes)
    variant: str = "gmc"        # Alg. 1, the appendix's "server_momentum" (Alg. 3) / "lr_in_residual"
                                # (Alg. 4), or the baseline "local_momentum" / "local_momentum_mfm"

    @property
    def k(self) -> int:
        return max(1, math.floor(self.ratio * self.d))


WORKLOADS = [
    Workload("mlp65k", d=65_536, K=4, compressor="topk", ratio=0.01, beta=0.9, eta=0.1,
             steps=10, iid_unit=True),
    Workload("resnet20", d=272_474, K=8, compressor="topk", ratio=0.01, beta=0.9, eta=0.1,
             steps=100, n_segments=20, noniid=0.02),
    Workload("resnet18", d=11_173_962, K=16, compressor="topk", ratio=0.001, beta=0.9,
             eta=0.05, steps=50, n_segments=62, laplace_frac=0.1, laplace_scale=5.0),
    Workload("resnet50", d=25_557_032, K=32, compressor="rbgs", ratio=0.01, beta=0.9,
             eta=0.1, steps=20, block=4096, lam=0.5, n_segments=161, noniid=0.02),
    # the resnet50 configuration with an independent block choice per worker and step
    Workload("resnet50_pw", d=25_557_032, K=32, compressor="rbgs", ratio=0.01, beta=0.9,
             eta=0.1, steps=20, block=4096, lam=0.5, per_worker=True, n_segments=161,
             noniid=0.02),
    Workload("vgg16", d=138_357_544, K=8, compressor="topk", ratio=0.001, beta=0.9,
             eta=0.01, steps=10, n_segments=32, big_segment=102_760_448,
             scale_lo=1e-4, scale_hi=1e-1, noniid=0.02),
    # the vgg16 configuration under the approximate top-s of Sec. 5.1 (s = d/1024)
    Workload("vgg16_approx", d=138_357_544, K=8, compressor="topk_approx", ratio=1 / 1024,
             beta=0.9, eta=0.01, steps=10, n_segments=32, big_segment=102_760_448,
             scale_lo=1e-4, scale_hi=1e-1, noniid=0.02),
    # the vgg16 configuration under the appendix's Alg. 3 and Alg. 4
    Workload("vgg16_alg3", d=138_357_544, K=8, compressor="topk", ratio=0.001, beta=0.9,
             eta=0.01, steps=10, n_segments=32, big_segment=102_760_448,
             scale_lo=1e-4, scale_hi=1e-1, noniid=0.02, variant="server_momentum"),
    Workload("vgg16_alg4", d=138_357_544, K=8, compressor="topk", ratio=0.001, beta=0.9,
             eta=0.01, steps=10, n_segments=32, big_segment=102_760_448,
             scale_lo=1e-4, scale_hi=1e-1, noniid=0.02, variant="lr_in_residual"),
    # the vgg16 and resnet50 configurations with bfloat16 gradient input
    Workload("vgg16_bf16", d=138_357_544, K=8, compressor="topk", ratio=0.001, beta=0.9,
             eta=0.01, steps=10, n_segments=32, big_segment=102_760_448,
             scale_lo=1e-4, scale_hi=1e-1, noniid=0.02, grad_dtype="bf16"),
    Workload("resnet50_bf16", d=25_557_032, K=32, compressor="rbgs", ratio=0.01, beta=0.9,
             eta=0.1, steps=20, block=4096, lam=0.5, n_segments=161, noniid=0.02,
             grad_dtype="bf16"),
    # and under the local-momentum baseline (DGC without / with momentum factor masking)
    Workload("vgg16_local", d=138_357_544, K=8, compressor="topk", ratio=0.001, beta=0.9,
             eta=0.01, steps=10, n_segments=32, big_segment=102_760_448,
             scale_lo=1e-4, scale_hi=1e-1, noniid=0.02, variant="local_momentum"),
    Workload("vgg16_local_mfm", d=138_357_544, K=8, compressor="topk", ratio=0.001, beta=0.9,
             eta=0.01, steps=10, n_segments=32, big_segment=102_760_448,
             scale_lo=1e-4, scale_hi=1e-1, noniid=0.02, variant="local_momentum_mfm"),
]


def workload(name_or_index) -> Workload:
    if isinstance(name_or_index, int):
        return WORKLOADS[name_or_index]
    for wl in WORKLOADS:
        if wl.name == name_or_index:
            return wl
    raise KeyError(name_or_index)


def _rng(seed: int, *stream: int) -> np.random.Generator:
    return np.random.Generator(np.random.Philox(np.random.SeedSequence([seed, *stream])))


def segment_sizes(wl: Workload, seed: int = 0) -> np.ndarray:
    """Layer segment sizes summing exactly to d (seeded cut points)."""
    if wl.iid_unit or wl.n_segments <= 1:
        return np.array([wl.d], np.int64)
    rng = _rng(seed, 101)
    n = wl.n_segments
    if wl.big_segment:
        rest = wl.d - wl.big_segment
        cuts = np.sort(rng.choice(rest - 1, size=n - 2, replace=False) + 1)
        small = np.diff(np.concatenate([[0], cuts, [rest]]))
        at = int(rng.integers(0, n))
        sizes = np.insert(small, at, wl.big_segment)
    else:
        cuts = np.sort(rng.choice(wl.d - 1, size=n - 1, replace=False) + 1)
        sizes = np.diff(np.concatenate([[0], cuts, [wl.d]]))
    assert sizes.sum() == wl.d and (sizes > 0).all()
    return sizes.astype(np.int64)


def segment_scales(wl: Workload, seed: int = 0) -> np.ndarray:
    """Per-segment gradient std, log-uniform on [scale_lo, scale_hi]."""
    n = len(segment_sizes(wl, seed))
    rng = _rng(seed, 102)
    lo, hi = math.log(wl.scale_lo), math.log(wl.scale_hi)
    return np.exp(rng.uniform(lo, hi, size=n)).astype(np.float32)


def element_scale(wl: Workload, seed: int = 0) -> np.ndarray:
    """Per-parameter gradient std (float32, length d)."""
    if wl.iid_unit:
        return np.ones(wl.d, np.float32)
    return np.repeat(segment_scales(wl, seed), segment_sizes(wl, seed)).astype(np.float32)


def init_params(d: int, seed: int = 0, std: float = 0.01) -> np.ndarray:
    """w_0 ~ N(0, std^2), float32."""
    return (_rng(seed, 7).standard_normal(d, dtype=np.float32) * np.float32(std)).astype(np.float32)


class NumpyGradients:
    """Host gradients g_t[K, d] (float32) for step t; same values on every call."""

    def __init__(self, wl: Workload, seed: int = 0, d: Optional[int] = None, K: Optional[int] = None):
        self.wl = wl
        self.seed = seed
        self.d = wl.d if d is None else d
        self.K = wl.K if K is None else K
        self.sigma = element_scale(wl, seed)[: self.d] if not wl.iid_unit else None
        self.mu = None
        if wl.noniid > 0:
            z = _rng(seed, 11).standard_normal((self.K, self.d), dtype=np.float32)
            self.mu = (z * (np.float32(wl.noniid) * self.sigma)).astype(np.float32)

    def __call__(self, t: int) -> np.ndarray:
        rng = _rng(self.seed, 1000 + t)
        z = rng.standard_normal((self.K, self.d), dtype=np.float32)
        if self.wl.iid_unit:
            return z
        if self.wl.laplace_frac > 0:
            heavy = rng.random((self.K, self.d), dtype=np.float32) < np.float32(self.wl.laplace_frac)
            lap = rng.laplace(0.0, self.wl.laplace_scale, size=(self.K, self.d)).astype(np.float32)
            z = np.where(heavy, lap, z)
        g = z * self.sigma
        if self.mu is not None:
            g = g + self.mu
        return g.astype(np.float32)


class TorchGradients:
    """Device gradients g_t[K, d] (float32 torch tensors), drawn with torch's RNG."""

    def __init__(self, wl: Workload, device, seed: int = 0):
        import torch
        self.torch = torch
        self.wl = wl
        self.device = device
        self.seed = seed
        self.sigma = None
        if not wl.iid_unit:
            self.sigma = torch.from_numpy(element_scale(wl, seed)).to(device)
        self.mu = None
        if wl.noniid > 0:
            gen = torch.Generator(device=device)
            gen.manual_seed(seed * 1_000_003 + 11)
            self.mu = torch.randn((wl.K, wl.d), generator=gen, device=device, dtype=torch.float32)
            self.mu.mul_(self.sigma * wl.noniid)

    def __call__(self, t: int, out=None):
        torch = self.torch
        wl = self.wl
        gen = torch.Generator(device=self.device)
        gen.manual_seed(self.seed * 1_000_003 + 1000 + t)
        if out is None:
            out = torch.empty((wl.K, wl.d), device=self.device, dtype=torch.float32)
        out.normal_(generator=gen)
        if wl.iid_unit:
            return out
        if wl.laplace_frac > 0:
            u = torch.rand((wl.K, wl.d), generator=gen, device=self.device) - 0.5
            # |u| < 1/2 keeps the inverse CDF finite (rand() can return exactly 0)
            mag = torch.clamp(u.abs(), max=0.5 - 2.0 ** -25)
            lap = -wl.laplace_scale * torch.sign(u) * torch.log1p(-2.0 * mag)
            del mag
            heavy = torch.rand((wl.K, wl.d), generator=gen, device=self.device) < wl.laplace_frac
            out.copy_(torch.where(heavy, lap, out))
            del u, lap, heavy
        out.mul_(self.sigma)
        if self.mu is not None:
            out.add_(self.mu)
        return out
