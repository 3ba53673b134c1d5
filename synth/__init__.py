"""Seeded synthetic inputs shaped like the paper's Wan2.1 workloads.

This module holds input generation only (no part of the method's arithmetic);
both the oracle side (tests) and the CUDA side (tests, bench) draw from it.

Recipe (stand-in for the paper's Wan2.1-T2V-1.3B generations, which need
model weights that are not available):
  * Q ~ N(0, 1) i.i.d. per element, fresh per segment and per denoising step.
  * K, V per latent frame follow an elementwise AR(1) process across frames,
    X_0 = Z_0, X_f = rho_f X_{f-1} + sqrt(1 - rho_f^2) Z_f, Z i.i.d. N(0, 1),
    so every frame has unit variance and neighbouring frames correlate by rho.
  * Independent streams for K, V, Q, each layer and each step; seed 0 default.
  * Values are drawn in fp32 and rounded to nearest even into the storage
    dtype (bf16 configs); the oracle then widens exactly those values to fp64.
Host generation (numpy PCG64) serves the small parity cases; device generation
(torch's CUDA generator, same recipe) serves the large configurations, and the
oracle consumes the generated values after they are copied back.
"""
from .inputs import (KIND_K, KIND_V, KIND_Q, host_rng, HostAR1, host_queries, round_to, DeviceAR1,
                     device_queries, rho_const, rho_drift)

__all__ = ["KIND_K", "KIND_V", "KIND_Q", "host_rng", "HostAR1", "host_queries", "round_to", "DeviceAR1",
           "device_queries", "rho_const", "rho_drift"]
