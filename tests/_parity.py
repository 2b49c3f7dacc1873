"""Shared helpers for the GPU parity tests: upload a workload, run the library
through its C-ABI binding, run the oracle on the same inputs, compare."""
from __future__ import annotations

import numpy as np
import torch

from oracle import flashslice_oracle as orc

# Tolerances of the comparison (per tensor):
#   fp32 inputs: normwise max relative error  max|gpu - ref| / max|ref| <= 1e-4
#   bf16 inputs: relative L2 error            ||gpu - ref||_2 / ||ref||_2 <= 1e-2
TOL_F32_MAXREL = 1e-4
TOL_BF16_RELL2 = 1e-2


def max_rel(a, ref):
    a = np.asarray(a, np.float64)
    ref = np.asarray(ref, np.float64)
    den = np.abs(ref).max()
    return float(np.abs(a - ref).max() / den) if den > 0 else float(np.abs(a).max())


def rel_l2(a, ref):
    a = np.asarray(a, np.float64)
    ref = np.asarray(ref, np.float64)
    den = np.linalg.norm(ref)
    return float(np.linalg.norm(a - ref) / den) if den > 0 else float(np.linalg.norm(a))


def error(a, ref, dtype):
    return max_rel(a, ref) if dtype == "f32" else rel_l2(a, ref)


def tol(dtype):
    return TOL_F32_MAXREL if dtype == "f32" else TOL_BF16_RELL2


def to_dev(arr, dtype, device="cuda"):
    t = torch.from_numpy(np.ascontiguousarray(arr))
    return t.to(device=device, dtype=torch.bfloat16 if dtype == "bf16" else torch.float32).contiguous()


def upload(wl, device="cuda"):
    dev = {
        "x_mid": to_dev(wl.x_mid, wl.dtype, device),
        "fx": to_dev(wl.fx, wl.dtype, device),
        "W_slice": to_dev(wl.W_slice, "f32", device),
        "bias": to_dev(wl.bias, "f32", device),
        "tau": to_dev(wl.tau, "f32", device),
        "M": to_dev(wl.M, "f32", device),
    }
    if wl.dout is not None:
        dev["dout"] = to_dev(wl.dout, wl.dtype, device)
    return dev


def host(t):
    return t.detach().float().cpu().numpy().astype(np.float64)


def gpu_forward(fs, wl, dev, coupling=None):
    c = coupling or fs.Coupling(wl.B, wl.N, wl.H, wl.d, wl.G,
                                torch.bfloat16 if wl.dtype == "bf16" else torch.float32, wl.eps,
                                backward=wl.dout is not None)
    c.forward(dev["x_mid"], dev["fx"], dev["W_slice"], dev["bias"], dev["tau"], dev["M"])
    return c


def oracle_forward(wl, heads=None, points=None):
    return orc.forward(wl.x_mid, wl.fx, wl.W_slice, wl.bias, wl.tau, wl.M, eps=wl.eps, heads=heads, points=points)


def oracle_backward(wl, heads=None):
    return orc.backward(wl.x_mid, wl.fx, wl.W_slice, wl.bias, wl.tau, wl.M, wl.dout, eps=wl.eps, heads=heads)


def lse_bound(wl, b, h, points, split=False):
    """Per-point bound on |lse_gpu - lse_exact| for head h of batch b at `points`,
    from the arithmetic of each path.
    * fp32 path: fp32 accumulation of the logits: 1e-4 absolute.
    * bf16 path (tensor cores): W' = W log2(e)/tau is rounded to bf16 (relative
      error <= 2^-8), or with split products (FS_DOT_BF16X2) rides as two bf16
      halves, hi + lo (residual <= 2^-16); x is bf16 already, exact; the bias
      rides as two halves (<= 2^-16). lse is a smooth maximum of the logits, so
      its error is at most the largest logit error of the point."""
    pts = np.asarray(points)
    if wl.dtype == "f32":
        return np.full(len(pts), 1e-4)
    Wp = np.abs(wl.W_slice[h].astype(np.float64)) * np.log2(np.e) / wl.tau[h]
    bp = np.abs(wl.bias[h].astype(np.float64)).max() * np.log2(np.e) / wl.tau[h]
    s = np.abs(wl.x_mid[b, pts, h, :].astype(np.float64)) @ Wp
    rel = 2.0 ** -16 if split else 2.0 ** -8
    return np.log(2.0) * (rel * s.max(axis=1) + 2.0 ** -16 * bp) + 1e-4
