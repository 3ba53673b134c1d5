"""Synthetic AR(1) K/V frames and Gaussian queries (see package docstring)."""
from __future__ import annotations

import math

import numpy as np
import torch

KIND_K, KIND_V, KIND_Q = 1, 2, 3


def host_rng(seed: int, kind: int, layer: int = 0, step: int = 0) -> np.random.Generator:
    """Independent PCG64 stream per (kind, layer, step)."""
    ss = np.random.SeedSequence(entropy=int(seed), spawn_key=(int(kind), int(layer), int(step)))
    return np.random.Generator(np.random.PCG64(ss))


def rho_const(rho: float):
    return lambda f: float(rho)


def rho_drift(rho0: float, rho1: float, n_frames: int):
    """rho drifting linearly from rho0 (frame 0) to rho1 (last frame)."""
    span = max(n_frames - 1, 1)
    return lambda f: float(rho0 + (rho1 - rho0) * min(f, span) / span)


class HostAR1:
    """fp32 AR(1) frames of a fixed shape on the host, one frame per call."""

    def __init__(self, shape, seed: int, kind: int, layer: int = 0, rho=rho_const(0.9)):
        self.shape = tuple(shape)
        self.rng = host_rng(seed, kind, layer)
        self.rho = rho
        self.f = 0
        self.x = None

    def next(self) -> np.ndarray:
        z = self.rng.standard_normal(self.shape, dtype=np.float32)
        if self.x is None:
            self.x = z
        else:
            r = np.float32(self.rho(self.f))
            self.x = r * self.x + np.float32(math.sqrt(max(0.0, 1.0 - float(r) * float(r)))) * z
        self.f += 1
        return self.x

    def frames(self, n: int) -> np.ndarray:
        return np.stack([self.next() for _ in range(n)])


def host_queries(shape, seed: int, layer: int = 0, step: int = 0) -> np.ndarray:
    return host_rng(seed, KIND_Q, layer, step).standard_normal(shape, dtype=np.float32)


def round_to(x, dtype: torch.dtype) -> torch.Tensor:
    """fp32 values -> storage dtype, round to nearest even (torch's cast)."""
    t = torch.as_tensor(np.ascontiguousarray(x, dtype=np.float32))
    return t.to(dtype)


class DeviceAR1:
    """The same AR(1) recipe generated on a CUDA device with torch's Philox generator.

    Holds the fp32 state of the process on the device; ``next()`` returns the
    next frame rounded into ``dtype``.  Values differ from HostAR1's (another
    generator); the oracle consumes them after they are copied back.
    """

    def __init__(self, shape, seed: int, kind: int, layer: int = 0, rho=rho_const(0.9),
                 dtype=torch.bfloat16, device="cuda"):
        self.shape = tuple(shape)
        self.gen = torch.Generator(device=device)
        self.gen.manual_seed((int(seed) * 1000003 + int(kind) * 7919 + int(layer) * 104729) & 0x7FFFFFFFFFFFFFFF)
        self.rho = rho
        self.dtype = dtype
        self.device = device
        self.f = 0
        self.x = None
        self.z = torch.empty(self.shape, dtype=torch.float32, device=device)

    def next(self) -> torch.Tensor:
        self.z.normal_(generator=self.gen)
        if self.x is None:
            self.x = self.z.clone()
        else:
            r = float(self.rho(self.f))
            self.x.mul_(r).add_(self.z, alpha=math.sqrt(max(0.0, 1.0 - r * r)))
        self.f += 1
        return self.x.to(self.dtype)


def device_queries(shape, seed: int, layer: int = 0, step: int = 0, dtype=torch.bfloat16, device="cuda"):
    g = torch.Generator(device=device)
    g.manual_seed((int(seed) * 1000003 + KIND_Q * 7919 + int(layer) * 104729 + int(step) * 15485863)
                  & 0x7FFFFFFFFFFFFFFF)
    return torch.randn(shape, generator=g, dtype=torch.float32, device=device).to(dtype)
