"""Seeded synthetic inputs for the slice -> mix -> deslice coupling.

Holds none of the method's arithmetic: only random draws, bf16 rounding of the
draws, and shapes.  Both the CUDA path and the CPU oracle consume these
arrays, so they see bit-identical inputs (bf16 values are stored as the exact
float32 they represent; the oracle upcasts them exactly to fp64).

The five named workloads reproduce the shapes and value distributions of the
paper's one-layer systems measurements (Appendix G, Table "one layer at large
slice counts": H = 8, D = 32, G up to 1024, N up to ~1M points), with synthetic
data standing in for the paper's CFD meshes, which are not available here:

  tiny_f32         B=1 N=4,096     G=32    fp32  forward
  surface_bf16     B=1 N=32,768    G=64    bf16  forward
  batched_bf16     B=4 N=262,144   G=256   bf16  forward (Gaussian-mixture x_mid)
  large_g_bf16     B=1 N=1,048,576 G=1024  bf16  forward
  train_bf16       B=2 N=524,288   G=512   bf16  forward + backward (mixture x_mid)

All use H=8 heads of width d=32 (C=256 channels, channel c = head c//32).
Random generator: numpy PCG64 seeded with 1000 + the workload's index (1..5).
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Optional

import numpy as np


def bf16_round(a: np.ndarray) -> np.ndarray:
    """Round float32 values to the nearest bf16 (ties to even); returns float32."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    u = a.view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) & 0xFFFF0000
    return u.astype(np.uint32).view(np.float32)


@dataclass
class Workload:
    name: str
    B: int
    N: int
    H: int
    d: int
    G: int
    dtype: str  # "f32" or "bf16"
    backward: bool
    x_mid: np.ndarray  # [B,N,H,d] float32 (bf16-exact values when dtype == "bf16")
    fx: np.ndarray  # [B,N,H,d]
    W_slice: np.ndarray  # [H,d,G] float32
    bias: np.ndarray  # [H,G] float32
    tau: np.ndarray  # [H] float32
    M: np.ndarray  # [H,G,G] float32
    dout: Optional[np.ndarray] = None  # [B,N,H,d] when backward
    eps: float = 1e-5
    recipe: str = ""
    extra: dict = field(default_factory=dict)

    @property
    def points(self) -> int:
        return self.B * self.N


def _normal(rng, shape, std=1.0):
    return (rng.standard_normal(size=shape, dtype=np.float32) * np.float32(std)).astype(np.float32)


def _gmm_points(rng, B, N, C, comps=16, mean_std=2.0, sigma=0.5):
    """Gaussian mixture in R^C: means ~ N(0, 4) per channel, isotropic sigma,
    uniform component weights, one component per (b, n), shared by all heads."""
    means = _normal(rng, (comps, C), mean_std)
    comp = rng.integers(0, comps, size=(B, N))
    x = means[comp]
    x += _normal(rng, (B, N, C), sigma)
    return x


def _mixer_identity_noise(rng, H, G, std=0.1):
    return (np.eye(G, dtype=np.float32)[None, :, :] + _normal(rng, (H, G, G), std)).astype(np.float32)


NAMED = ("tiny_f32", "surface_bf16", "batched_bf16", "large_g_bf16", "train_bf16")


def make_named(name: str, n_override: Optional[int] = None, g_override: Optional[int] = None,
               dtype_override: Optional[str] = None) -> Workload:
    """One of the five named workloads; `n_override` changes N, `g_override` the slot
    count G and `dtype_override` the input dtype ("f32" or "bf16"; same recipe
    otherwise)."""
    idx = NAMED.index(name) + 1
    rng = np.random.Generator(np.random.PCG64(1000 + idx))
    H, d = 8, 32
    C = H * d
    if name == "tiny_f32":
        B, N, G, dtype, bwd = 1, 4096, 32, "f32", False
    elif name == "surface_bf16":
        B, N, G, dtype, bwd = 1, 32768, 64, "bf16", False
    elif name == "batched_bf16":
        B, N, G, dtype, bwd = 4, 262144, 256, "bf16", False
    elif name == "large_g_bf16":
        B, N, G, dtype, bwd = 1, 1048576, 1024, "bf16", False
    else:
        B, N, G, dtype, bwd = 2, 524288, 512, "bf16", True
    if n_override is not None:
        N = int(n_override)
    if g_override is not None:
        G = int(g_override)
    if dtype_override is not None:
        if dtype_override not in ("f32", "bf16"):
            raise ValueError(f"dtype_override must be 'f32' or 'bf16', got {dtype_override!r}")
        dtype = dtype_override
    mixture = name in ("batched_bf16", "train_bf16")
    if mixture:
        x = _gmm_points(rng, B, N, C).reshape(B, N, H, d)
        recipe_x = "x_mid ~ 16-component Gaussian mixture (means N(0,4), sigma 0.5)"
    else:
        x = _normal(rng, (B, N, H, d))
        recipe_x = "x_mid ~ N(0,1)"
    fx = _normal(rng, (B, N, H, d))
    W = _normal(rng, (H, d, G), 1.0 / np.sqrt(d))
    bias = np.zeros((H, G), np.float32)
    if name == "surface_bf16":
        tau = rng.uniform(0.3, 1.0, size=H).astype(np.float32)
        M = _normal(rng, (H, G, G), 1.0 / np.sqrt(G))
        recipe_m = "tau ~ U[0.3,1]; M ~ N(0,1/G)"
    else:
        tau = np.full(H, 0.5, np.float32)
        M = _mixer_identity_noise(rng, H, G)
        recipe_m = "tau = 0.5; M = I + N(0,0.01)"
    dout = _normal(rng, (B, N, H, d)) if bwd else None
    if dtype == "bf16":
        x = bf16_round(x)
        fx = bf16_round(fx)
        if dout is not None:
            dout = bf16_round(dout)
    recipe = (f"{recipe_x}; fx ~ N(0,1); W ~ N(0,1/d); bias = 0; {recipe_m}"
              + ("; dout ~ N(0,1)" if bwd else "") + f"; PCG64 seed {1000 + idx}")
    return Workload(name, B, N, H, d, G, dtype, bwd, x, fx, W, bias, tau, M, dout, 1e-5, recipe)


def make_case(B, N, H, d, G, dtype="f32", seed=0, bias_std=0.1, tau=None, x_std=1.0,
              mixture=False, backward=True, eps=1e-5, m_std=0.1) -> Workload:
    """A small random case for parity tests (random bias so dbias is exercised).

    tau: None draws tau_h ~ U[0.3, 1.0]; a float fixes every head.
    """
    rng = np.random.Generator(np.random.PCG64(seed))
    if mixture:
        x = _gmm_points(rng, B, N, H * d).reshape(B, N, H, d)
    else:
        x = _normal(rng, (B, N, H, d), x_std)
    fx = _normal(rng, (B, N, H, d))
    W = _normal(rng, (H, d, G), 1.0 / np.sqrt(d))
    bias = _normal(rng, (H, G), bias_std)
    if tau is None:
        t = rng.uniform(0.3, 1.0, size=H).astype(np.float32)
    else:
        t = np.full(H, tau, np.float32)
    M = _mixer_identity_noise(rng, H, G, m_std)
    dout = _normal(rng, (B, N, H, d)) if backward else None
    if dtype == "bf16":
        x = bf16_round(x)
        fx = bf16_round(fx)
        if dout is not None:
            dout = bf16_round(dout)
    return Workload(f"case_B{B}_N{N}_H{H}_d{d}_G{G}_{dtype}", B, N, H, d, G, dtype, backward,
                    x, fx, W, bias, t, M, dout, eps, "make_case")
