"""GPU parity at large slice counts against the fp64 oracle: G beyond 1024 up to
the header's limit of 4096 (forward and backward, fp32 and bf16 inputs, every
supported head width; the forward on the fp32 SIMT kernels, the bf16 d = 32
backward on the tensor cores over slot ranges), the bf16 backward beyond G = 640
after a tensor-core forward, and fp32 inputs at G = 768 and 1024 (the fp32
tensor-core forward, its deslice over slot ranges past 512 slots).

Tolerances (tests/_parity.py): fp32 inputs normwise max relative error <= 1e-4
per tensor; bf16 inputs relative L2 error <= 1e-2 per tensor.
"""
import numpy as np
import pytest
import torch

from paper_2609_32525_gb300.workloads import make_case

from _parity import error, gpu_forward, host, oracle_backward, oracle_forward, tol, upload

pytestmark = pytest.mark.gpu

# (B, N, H, d, G): G past the tensor-core limit, a ragged point count, B > 1.
LARGE_G = [
    (1, 301, 2, 32, 1500),
    (2, 129, 1, 16, 2049),
    (1, 200, 2, 64, 3001),
    (1, 257, 1, 32, 4096),
]


def _check(name, got, ref, dtype):
    e = error(got, ref, dtype)
    assert e <= tol(dtype), f"{name}: error {e:.3e} > {tol(dtype):.0e}"


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("shp", LARGE_G, ids=lambda s: "B{}N{}H{}d{}G{}".format(*s))
def test_large_g_forward_and_backward(lib, shp, dtype):
    B, N, H, d, G = shp
    wl = make_case(B, N, H, d, G, dtype=dtype, seed=1300 + G + N, backward=True)
    dev = upload(wl)
    c = gpu_forward(lib, wl, dev)
    assert lib.path_for_shape(c.shape) == 0
    assert lib.backward_path_for_shape(c.shape) == (1 if dtype == "bf16" and d == 32 else 0)
    g = c.backward(dev["x_mid"], dev["fx"], dev["W_slice"], dev["bias"], dev["tau"], dev["M"], dev["dout"])
    torch.cuda.synchronize()
    assert c.device_status() == lib.FS_OK
    ref = oracle_forward(wl)
    for k in ("tokens", "wsum", "tokens_mixed", "out"):
        _check(k, host(getattr(c, k)), ref[k], dtype)
    rb = oracle_backward(wl)
    for k in ("dx_mid", "dfx", "dW", "dbias", "dtau", "dM"):
        _check(k, host(g[k]), rb[k], dtype)
    _check("d_tokens_mixed", host(c.d_tokens_mixed), rb["d_tokens_mixed"], dtype)


@pytest.mark.parametrize("G", [768, 1024])
def test_bf16_backward_over_slot_ranges(lib, G):
    """bf16, d = 32, G > 640: the forward on tensor cores, the backward on tensor
    cores over slot ranges (with split-product statistics recomputed)."""
    wl = make_case(1, 1500, 2, 32, G, dtype="bf16", seed=1400 + G, backward=True)
    dev = upload(wl)
    c = gpu_forward(lib, wl, dev)
    assert lib.path_for_shape(c.shape) == 1 and lib.backward_path_for_shape(c.shape) == 1
    g = c.backward(dev["x_mid"], dev["fx"], dev["W_slice"], dev["bias"], dev["tau"], dev["M"], dev["dout"])
    torch.cuda.synchronize()
    assert c.device_status() == lib.FS_OK
    rb = oracle_backward(wl)
    for k in ("dx_mid", "dfx", "dW", "dbias", "dtau", "dM"):
        _check(k, host(g[k]), rb[k], "bf16")


@pytest.mark.parametrize("G", [768, 1024])
def test_fp32_above_512_slots_on_tensor_cores(lib, G):
    """fp32 inputs with B*N*H*G >= 2^24 at G = 768 and 1024: the tensor-core
    forward, its deslice over slot ranges, at the fp32 bar."""
    N = 3000
    assert N * 8 * G >= 1 << 24
    wl = make_case(1, N, 8, 32, G, dtype="f32", seed=1500 + G, backward=False)
    dev = upload(wl)
    c = gpu_forward(lib, wl, dev)
    assert lib.path_for_shape(c.shape) == 1
    torch.cuda.synchronize()
    assert c.device_status() == lib.FS_OK
    ref = oracle_forward(wl)
    for k in ("tokens", "wsum", "tokens_mixed", "out"):
        _check(k, host(getattr(c, k)), ref[k], "f32")
    assert np.abs(host(c.lse) - ref["lse"].transpose(0, 2, 1)).max() < 1e-4
