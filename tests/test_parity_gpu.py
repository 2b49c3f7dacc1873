"""GPU parity: the CUDA library (through its C ABI) against the fp64 oracle on
the same seeded inputs, element by element.

Tolerances (tests/_parity.py): fp32 inputs max relative error <= 1e-4 per
tensor (normwise); bf16 inputs relative L2 error <= 1e-2 per tensor.
"""
import numpy as np
import pytest
import torch

from paper_2609_32525_gb300.workloads import make_case

from _parity import error, gpu_forward, host, oracle_backward, oracle_forward, tol, upload

pytestmark = pytest.mark.gpu

# (B, N, H, d, G): slot counts 1, 3, 48, 100, 130 (non powers of two), point
# counts that are not multiples of any tile, B > 1, every supported d.
SMALL = [
    (1, 1, 1, 16, 1),
    (2, 300, 2, 32, 3),
    (1, 1000, 3, 16, 48),
    (2, 513, 2, 32, 100),
    (1, 777, 2, 64, 130),
    (1, 4096, 8, 32, 32),
    (1, 3000, 2, 32, 256),
    (1, 2500, 1, 32, 1024),
]


def _check(name, got, ref, dtype, extra=""):
    e = error(got, ref, dtype)
    assert e <= tol(dtype), f"{name}: error {e:.3e} > {tol(dtype):.0e} {extra}"
    return e


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("shp", SMALL, ids=lambda s: "B{}N{}H{}d{}G{}".format(*s))
def test_forward_small(lib, shp, dtype):
    B, N, H, d, G = shp
    wl = make_case(B, N, H, d, G, dtype=dtype, seed=100 + G + N, backward=False)
    dev = upload(wl)
    c = gpu_forward(lib, wl, dev)
    torch.cuda.synchronize()
    assert c.device_status() == lib.FS_OK
    ref = oracle_forward(wl)
    _check("tokens", host(c.tokens), ref["tokens"], dtype)
    _check("wsum", host(c.wsum), ref["wsum"], dtype)
    _check("tokens_mixed", host(c.tokens_mixed), ref["tokens_mixed"], dtype)
    _check("out", host(c.out), ref["out"], dtype)
    # lse is a per-point statistic: absolute error in nats, fp32 accumulate.
    assert np.abs(host(c.lse) - ref["lse"].transpose(0, 2, 1)).max() < (1e-4 if dtype == "f32" else 5e-2)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("shp", SMALL[:6], ids=lambda s: "B{}N{}H{}d{}G{}".format(*s))
def test_backward_small(lib, shp, dtype):
    B, N, H, d, G = shp
    wl = make_case(B, N, H, d, G, dtype=dtype, seed=200 + G + N, backward=True)
    dev = upload(wl)
    c = gpu_forward(lib, wl, dev)
    g = c.backward(dev["x_mid"], dev["fx"], dev["W_slice"], dev["bias"], dev["tau"], dev["M"], dev["dout"])
    torch.cuda.synchronize()
    assert c.device_status() == lib.FS_OK
    ref = oracle_backward(wl)
    for k in ("dx_mid", "dfx", "dW", "dbias", "dtau", "dM"):
        _check(k, host(g[k]), ref[k], dtype)
    _check("d_tokens_mixed", host(c.d_tokens_mixed), ref["d_tokens_mixed"], dtype)


def test_unnormalised_partials_and_finalize(lib):
    wl = make_case(2, 700, 2, 32, 40, dtype="bf16", seed=7, backward=False)
    dev = upload(wl)
    s = lib.shape_of(dev["x_mid"], wl.G, wl.eps)
    ws = lib.workspace(s, lib.FS_OP_SLICE_FWD)
    f32 = dict(dtype=torch.float32, device="cuda")
    U = torch.empty(2, 2, 40, 32, **f32)
    S = torch.empty(2, 2, 40, **f32)
    Z = torch.empty(2, 2, 40, 32, **f32)
    lib.fs_slice_fwd(s, dev["x_mid"], dev["fx"], dev["W_slice"], dev["bias"], dev["tau"], U, S, None, False, ws)
    lib.fs_slice_fwd(s, dev["x_mid"], dev["fx"], dev["W_slice"], dev["bias"], dev["tau"], Z, S, None, True, ws)
    Uf = U.clone()
    lib.fs_slice_finalize(s, Uf, S)
    torch.cuda.synchronize()
    np.testing.assert_allclose(host(Uf), host(Z), rtol=1e-6, atol=1e-7)
    ref = oracle_forward(wl)
    assert error(host(U) / (host(S)[..., None] + wl.eps), ref["tokens"], "bf16") < 1e-2


def test_deslice_without_statistics(lib):
    """lse = NULL: the deslice computes the statistics itself."""
    wl = make_case(1, 900, 2, 32, 70, dtype="f32", seed=8, backward=False)
    dev = upload(wl)
    ref = oracle_forward(wl)
    s = lib.shape_of(dev["x_mid"], wl.G, wl.eps)
    tm = torch.from_numpy(ref["tokens_mixed"].astype(np.float32)).cuda()
    out = torch.empty_like(dev["x_mid"])
    ws = lib.workspace(s, lib.FS_OP_DESLICE_FWD)
    lib.fs_deslice_fwd(s, dev["x_mid"], dev["W_slice"], dev["bias"], dev["tau"], tm, None, out, ws)
    torch.cuda.synchronize()
    _check("out", host(out), ref["out"], "f32")


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_bitwise_determinism(lib, dtype):
    wl = make_case(2, 5000, 4, 32, 200, dtype=dtype, seed=9, backward=True)
    dev = upload(wl)
    res = []
    for _ in range(2):
        c = gpu_forward(lib, wl, dev)
        g = c.backward(dev["x_mid"], dev["fx"], dev["W_slice"], dev["bias"], dev["tau"], dev["M"], dev["dout"])
        torch.cuda.synchronize()
        res.append([t.clone() for t in (c.tokens, c.out, c.lse, g["dx_mid"], g["dfx"], g["dW"], g["dbias"],
                                        g["dtau"], g["dM"])])
    for a, b in zip(*res):
        assert torch.equal(a.view(torch.uint8) if a.dtype != torch.bfloat16 else a.view(torch.int16),
                           b.view(torch.uint8) if b.dtype != torch.bfloat16 else b.view(torch.int16))


def test_bad_tau_sets_device_status(lib):
    wl = make_case(1, 300, 2, 32, 16, dtype="f32", seed=10, backward=False)
    dev = upload(wl)
    dev["tau"][1] = -0.5
    c = gpu_forward(lib, wl, dev)
    torch.cuda.synchronize()
    assert lib.fs_device_status(c.ws_slice) == lib.FS_ERR_BAD_TAU
    dev["tau"][1] = 0.5
    c = gpu_forward(lib, wl, dev, c)
    assert lib.fs_device_status(c.ws_slice) == lib.FS_OK


def test_uniform_weights_on_gpu(lib):
    """W = 0, bias = 0: every token is the global mean sum f / (N + G eps)."""
    wl = make_case(1, 4000, 2, 32, 64, dtype="f32", seed=11, backward=False)
    wl.W_slice[:] = 0
    wl.bias[:] = 0
    dev = upload(wl)
    c = gpu_forward(lib, wl, dev)
    torch.cuda.synchronize()
    mean = wl.fx[0].astype(np.float64).sum(axis=0) / (wl.N + wl.G * wl.eps)  # [H, d]
    for h in range(2):
        np.testing.assert_allclose(host(c.tokens)[0, h], np.broadcast_to(mean[h], (64, 32)), rtol=2e-5, atol=2e-6)
