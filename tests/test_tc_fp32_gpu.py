"""GPU parity of the tensor-core forward for fp32 inputs (d = 32, G <= 1024,
B*N*H*G >= 2^24; smaller fp32 problems keep the exact SIMT kernels): every
operand as two bf16 halves (x, fx, W' = W log2(e)/tau, the weights, z'), the
paper's three-product level for fp32 data (App. G.2 dot levels); past 512 slots
the deslice runs over slot ranges whose fp32 outputs add up.  Against the fp64
oracle at the fp32 bar: normwise max relative error <= 1e-4 for tokens, wsum,
tokens_mixed, out and lse.  The backward of these shapes runs on the fp32 SIMT
kernels with exact fp32 statistics; it is checked too.
"""
import numpy as np
import pytest
import torch

from oracle import flashslice_oracle as orc
from paper_2609_32525_gb300.workloads import make_case

from _parity import host, max_rel, upload

pytestmark = pytest.mark.gpu

# G = 640, 700 and 1024 run the deslice over slot ranges: 384 + 256, 384 + 316 and
# 2 x 512.
SHAPES = [(1, 20001, 8, 128), (1, 33000, 8, 100), (2, 9000, 8, 256), (1, 5000, 8, 512), (1, 70000, 8, 32),
          (1, 4000, 8, 640), (1, 3001, 8, 700), (1, 2500, 8, 1024)]
TOL = 1e-4


@pytest.mark.parametrize("shp", SHAPES, ids=lambda s: "B{}N{}H{}G{}".format(*s))
def test_fp32_tensor_core_forward(lib, shp):
    B, N, H, G = shp
    wl = make_case(B, N, H, 32, G, dtype="f32", seed=800 + N + G, backward=False)
    dev = upload(wl)
    c = lib.Coupling(B, N, H, 32, G, torch.float32, wl.eps)
    assert lib.path_for_shape(c.shape) == 1
    c.forward(dev["x_mid"], dev["fx"], dev["W_slice"], dev["bias"], dev["tau"], dev["M"])
    torch.cuda.synchronize()
    assert c.device_status() == lib.FS_OK
    ref = orc.forward(wl.x_mid, wl.fx, wl.W_slice, wl.bias, wl.tau, wl.M, eps=wl.eps)
    errs = {"tokens": max_rel(host(c.tokens), ref["tokens"]), "wsum": max_rel(host(c.wsum), ref["wsum"]),
            "tokens_mixed": max_rel(host(c.tokens_mixed), ref["tokens_mixed"]),
            "out": max_rel(host(c.out), ref["out"]),
            "lse": max_rel(host(c.lse), ref["lse"].transpose(0, 2, 1))}
    print(shp, " ".join("{}={:.2e}".format(k, e) for k, e in errs.items()))
    bad = {k: e for k, e in errs.items() if not e <= TOL}
    assert not bad, {k: "{:.2e}".format(e) for k, e in bad.items()}


def test_small_fp32_problems_keep_the_simt_kernels(lib):
    assert lib.path_for_shape(lib.make_shape(1, 4096, 8, 32, 32, lib.FS_F32)) == 0
    assert lib.path_for_shape(lib.make_shape(1, 70000, 8, 32, 32, lib.FS_F32)) == 1
    assert lib.path_for_shape(lib.make_shape(1, 70000, 8, 32, 640, lib.FS_F32)) == 1
    assert lib.path_for_shape(lib.make_shape(1, 70000, 8, 32, 1024, lib.FS_F32)) == 1
    assert lib.path_for_shape(lib.make_shape(1, 70000, 8, 32, 1025, lib.FS_F32)) == 0


@pytest.mark.parametrize("G", [256, 512, 1024])
def test_fp32_backward_after_tensor_core_forward(lib, G):
    """The fp32 coupling's whole backward (fs_coupling_bwd on the fused SIMT kernels,
    exact fp32 statistics) after the tensor-core forward, at the fp32 bar."""
    N = 5000 if G == 256 else 3000
    wl = make_case(2, N, 8, 32, G, dtype="f32", seed=810 + G, backward=True)
    dev = upload(wl)
    c = lib.Coupling(wl.B, wl.N, wl.H, 32, wl.G, torch.float32, wl.eps, backward=True)
    assert lib.path_for_shape(c.shape) == 1 and lib.backward_path_for_shape(c.shape) == 0
    c.forward(dev["x_mid"], dev["fx"], dev["W_slice"], dev["bias"], dev["tau"], dev["M"])
    g = c.backward(dev["x_mid"], dev["fx"], dev["W_slice"], dev["bias"], dev["tau"], dev["M"], dev["dout"])
    torch.cuda.synchronize()
    assert c.device_status() == lib.FS_OK
    ref = orc.backward(wl.x_mid, wl.fx, wl.W_slice, wl.bias, wl.tau, wl.M, wl.dout, eps=wl.eps)
    errs = {k: max_rel(host(g[k]), ref[k]) for k in ("dx_mid", "dfx", "dW", "dbias", "dtau", "dM")}
    print("fp32 backward G={}".format(G), " ".join("{}={:.2e}".format(k, e) for k, e in errs.items()))
    bad = {k: e for k, e in errs.items() if not e <= TOL}
    assert not bad, {k: "{:.2e}".format(e) for k, e in bad.items()}


def test_fp32_tensor_core_forward_long_point_ranges(lib):
    """fp32 inputs over long point ranges: at N = 786,432, B*H = 8 and two 128-slot blocks,
    each slice CTA reduces ~41,000 points (19 point splits), ~320 tiles into each
    tensor-core accumulator chain.  One chain over the whole range loses ~2^-25 of its
    running sum per K step, always towards zero, about 1e-4 relative at this length;
    the slice moves its accumulators into fp32 registers every few tiles instead.  One
    head is checked over all points (tokens, wsum, tokens_mixed) and a point sample
    (out, lse) at the fp32 bar."""
    B, N, H, G = 1, 786432, 8, 256
    wl = make_case(B, N, H, 32, G, dtype="f32", seed=821, backward=False)
    dev = upload(wl)
    c = lib.Coupling(B, N, H, 32, G, torch.float32, wl.eps)
    assert lib.path_for_shape(c.shape) == 1
    c.forward(dev["x_mid"], dev["fx"], dev["W_slice"], dev["bias"], dev["tau"], dev["M"])
    torch.cuda.synchronize()
    assert c.device_status() == lib.FS_OK
    h = 5
    rng = np.random.default_rng(822)
    pts = np.unique(np.concatenate([np.arange(64), np.arange(N - 64, N), rng.integers(0, N, size=4096)]))
    ref = orc.forward(wl.x_mid, wl.fx, wl.W_slice, wl.bias, wl.tau, wl.M, eps=wl.eps, heads=[h], points=pts)
    errs = {"tokens": max_rel(host(c.tokens)[:, h], ref["tokens"][:, h]),
            "wsum": max_rel(host(c.wsum)[:, h], ref["wsum"][:, h]),
            "tokens_mixed": max_rel(host(c.tokens_mixed)[:, h], ref["tokens_mixed"][:, h]),
            "out": max_rel(host(c.out)[:, pts][:, :, h], ref["out"][:, pts][:, :, h]),
            "lse": max_rel(host(c.lse)[:, h, pts], ref["lse"][:, pts, h])}
    print("long ranges", " ".join("{}={:.2e}".format(k, e) for k, e in errs.items()))
    bad = {k: e for k, e in errs.items() if not e <= TOL}
    assert not bad, {k: "{:.2e}".format(e) for k, e in bad.items()}
