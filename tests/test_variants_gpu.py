"""The coupling variants of Sec. 3 (the variants table) through the C ABI, against
the fp64 oracle:

* Untied: the deslice gets its own projection and temperature (W', beta', tau').
  fs_deslice_fwd and fs_deslice_bwd take them with lse = NULL (they compute the
  statistics of the deslice weights themselves); the slice keeps (W, beta, tau).
  Every output and gradient, both weight sets' gradients separately.
* FrozenSlice: a later layer slices its own features fx2 with the layer-1 logits
  input, weights and statistics: fs_slice_fwd_lse with the layer-1 lse, against the
  oracle's slice of fx2 with the layer-1 weights, and against fs_slice_fwd.

Shapes: tensor-core bf16 (d = 32; G = 256 and a padded G = 100), the fp32 tensor-core
path (d = 32, G = 128, B*N*H*G >= 2^24: split bf16 halves) and SIMT (fp32, d = 16).
Tolerances as everywhere: fp32 normwise max relative 1e-4; bf16 relative L2 1e-2.
"""
import numpy as np
import pytest
import torch

from oracle import flashslice_oracle as orc
from paper_2609_32525_gb300.workloads import make_case

from _parity import error, host, tol, upload

pytestmark = pytest.mark.gpu

CASES = [(2, 1500, 2, 32, 256, "bf16"), (1, 900, 2, 32, 100, "bf16"), (1, 70000, 2, 32, 128, "f32"),
         (2, 700, 2, 16, 40, "f32")]
IDS = ["tc-G256", "tc-G100-padded", "tc-f32-split", "simt-f32"]


def _f32(a):
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).cuda()


def _check(name, got, ref, dtype):
    e = error(got, ref, dtype)
    assert e <= tol(dtype), f"{name}: error {e:.3e} > {tol(dtype):.0e}"


@pytest.mark.parametrize("case", CASES, ids=IDS)
def test_untied_forward_and_backward(lib, case):
    B, N, H, d, G, dt = case
    wl = make_case(B, N, H, d, G, dtype=dt, seed=900 + G, backward=True)
    w2 = make_case(B, N, H, d, G, dtype=dt, seed=901 + G, backward=False)  # the deslice's own weights
    dev = upload(wl)
    W2, b2, t2 = _f32(w2.W_slice), _f32(w2.bias), _f32(w2.tau)
    s = lib.shape_of(dev["x_mid"], G, wl.eps, dot=lib.FS_DOT_BF16X2)
    f32 = dict(dtype=torch.float32, device="cuda")
    pdt = dev["x_mid"].dtype
    tokens, wsum, lse = (torch.empty(B, H, G, d, **f32), torch.empty(B, H, G, **f32), torch.empty(B, H, N, **f32))
    tm, out = torch.empty(B, H, G, d, **f32), torch.empty(B, N, H, d, dtype=pdt, device="cuda")
    ws_s, ws_d = lib.workspace(s, lib.FS_OP_SLICE_FWD), lib.workspace(s, lib.FS_OP_DESLICE_FWD)
    lib.fs_slice_fwd(s, dev["x_mid"], dev["fx"], dev["W_slice"], dev["bias"], dev["tau"], tokens, wsum, lse, True,
                     ws_s)
    lib.fs_mix(s, dev["M"], tokens, tm)
    lib.fs_deslice_fwd(s, dev["x_mid"], W2, b2, t2, tm, None, out, ws_d)
    # backward: the deslice's weights (lse = NULL), then the slice's
    dzm, dz = torch.empty(B, H, G, d, **f32), torch.empty(B, H, G, d, **f32)
    dx = torch.empty(B, N, H, d, dtype=pdt, device="cuda")
    dfx = torch.empty_like(dx)
    dW2, db2, dt2 = torch.empty(H, d, G, **f32), torch.empty(H, G, **f32), torch.empty(H, **f32)
    # the slice's call adds (accumulate = 1: dx onto the deslice's); its own weights' gradients start at zero
    dW1, db1, dt1 = torch.zeros(H, d, G, **f32), torch.zeros(H, G, **f32), torch.zeros(H, **f32)
    dM = torch.empty(H, G, G, **f32)
    ws_db, ws_sb = lib.workspace(s, lib.FS_OP_DESLICE_BWD), lib.workspace(s, lib.FS_OP_SLICE_BWD)
    lib.fs_deslice_bwd(s, dev["x_mid"], W2, b2, t2, tm, None, dev["dout"], dzm, dx, dW2, db2, dt2, False, ws_db)
    lib.fs_mix_bwd(s, dev["M"], tokens, dzm, dz, dM)
    lib.fs_slice_bwd(s, dev["x_mid"], dev["fx"], dev["W_slice"], dev["bias"], dev["tau"], tokens, wsum, lse, dz, dx,
                     dfx, dW1, db1, dt1, True, ws_sb)
    torch.cuda.synchronize()
    for w in (ws_s, ws_d, ws_db, ws_sb):
        assert lib.fs_device_status(w) == lib.FS_OK

    ref_s = orc.slice_fwd(wl.x_mid, wl.fx, wl.W_slice, wl.bias, wl.tau, eps=wl.eps)
    ref_tm = orc.mix(wl.M, ref_s["tokens"])
    ref_out = orc.deslice_fwd(wl.x_mid, w2.W_slice, w2.bias, w2.tau, ref_tm)
    rd = orc.deslice_bwd(wl.x_mid, w2.W_slice, w2.bias, w2.tau, ref_tm, wl.dout)
    rm = orc.mix_bwd(wl.M, ref_s["tokens"], rd["d_tokens_mixed"])
    rs = orc.slice_bwd(wl.x_mid, wl.fx, wl.W_slice, wl.bias, wl.tau, ref_s["tokens"], ref_s["wsum"], rm["d_tokens"],
                       eps=wl.eps)
    _check("out", host(out), ref_out, dt)
    _check("tokens", host(tokens), ref_s["tokens"], dt)
    _check("d_tokens_mixed", host(dzm), rd["d_tokens_mixed"], dt)
    _check("dM", host(dM), rm["dM"], dt)
    _check("dx_mid", host(dx), rd["dx_mid"] + rs["dx_mid"], dt)
    _check("dfx", host(dfx), rs["dfx"], dt)
    for name, got, ref in (("dW (deslice)", dW2, rd["dW"]), ("dbias (deslice)", db2, rd["dbias"]),
                           ("dtau (deslice)", dt2, rd["dtau"]), ("dW (slice)", dW1, rs["dW"]),
                           ("dbias (slice)", db1, rs["dbias"]), ("dtau (slice)", dt1, rs["dtau"])):
        _check(name, host(got), ref, dt)


@pytest.mark.parametrize("case", CASES, ids=IDS)
def test_frozen_slice_with_layer1_statistics(lib, case):
    B, N, H, d, G, dt = case
    wl = make_case(B, N, H, d, G, dtype=dt, seed=950 + G, backward=False)
    layer2 = make_case(B, N, H, d, G, dtype=dt, seed=951 + G, backward=False)  # its fx: the later layer's features
    dev = upload(wl)
    pdt = dev["x_mid"].dtype
    fx2 = torch.from_numpy(np.ascontiguousarray(layer2.fx)).to("cuda", pdt)
    s = lib.shape_of(dev["x_mid"], G, wl.eps)
    f32 = dict(dtype=torch.float32, device="cuda")
    ws = lib.workspace(s, lib.FS_OP_SLICE_FWD)
    tok1, ws1, lse1 = torch.empty(B, H, G, d, **f32), torch.empty(B, H, G, **f32), torch.empty(B, H, N, **f32)
    lib.fs_slice_fwd(s, dev["x_mid"], dev["fx"], dev["W_slice"], dev["bias"], dev["tau"], tok1, ws1, lse1, True, ws)
    tok2, wsum2 = torch.full_like(tok1, float("nan")), torch.full_like(ws1, float("nan"))
    lib.fs_slice_fwd_lse(s, dev["x_mid"], fx2, dev["W_slice"], dev["bias"], dev["tau"], lse1, tok2, wsum2, True, ws)
    tok2b, wsum2b = torch.empty_like(tok1), torch.empty_like(ws1)
    lib.fs_slice_fwd(s, dev["x_mid"], fx2, dev["W_slice"], dev["bias"], dev["tau"], tok2b, wsum2b, None, True, ws)
    torch.cuda.synchronize()
    assert lib.fs_device_status(ws) == lib.FS_OK
    ref = orc.slice_fwd(wl.x_mid, layer2.fx, wl.W_slice, wl.bias, wl.tau, eps=wl.eps)
    _check("tokens", host(tok2), ref["tokens"], dt)
    _check("wsum", host(wsum2), ref["wsum"], dt)
    # the weight sums do not depend on fx: the same as layer 1's
    _check("wsum vs layer 1", host(wsum2), host(ws1), dt)
    _check("tokens vs fs_slice_fwd", host(tok2), host(tok2b), dt)


@pytest.mark.parametrize("case", CASES, ids=IDS)
def test_stats_alone_matches_the_slice_call(lib, case):
    """fs_stats writes the same lse as fs_slice_fwd (the same kernels), and
    fs_stats + fs_slice_fwd_lse gives the same tokens as fs_slice_fwd."""
    B, N, H, d, G, dt = case
    wl = make_case(B, N, H, d, G, dtype=dt, seed=960 + G, backward=False)
    dev = upload(wl)
    s = lib.shape_of(dev["x_mid"], G, wl.eps)
    f32 = dict(dtype=torch.float32, device="cuda")
    ws, ws_st = lib.workspace(s, lib.FS_OP_SLICE_FWD), lib.workspace(s, lib.FS_OP_STATS)
    tok, wsum, lse = torch.empty(B, H, G, d, **f32), torch.empty(B, H, G, **f32), torch.empty(B, H, N, **f32)
    lib.fs_slice_fwd(s, dev["x_mid"], dev["fx"], dev["W_slice"], dev["bias"], dev["tau"], tok, wsum, lse, True, ws)
    lse2 = torch.full_like(lse, float("nan"))
    lib.fs_stats(s, dev["x_mid"], dev["W_slice"], dev["bias"], dev["tau"], lse2, ws_st)
    tok2, wsum2 = torch.empty_like(tok), torch.empty_like(wsum)
    lib.fs_slice_fwd_lse(s, dev["x_mid"], dev["fx"], dev["W_slice"], dev["bias"], dev["tau"], lse2, tok2, wsum2, True,
                         ws)
    torch.cuda.synchronize()
    assert lib.fs_device_status(ws_st) == lib.FS_OK and lib.fs_device_status(ws) == lib.FS_OK
    assert torch.equal(lse, lse2)
    _check("tokens", host(tok2), host(tok), dt)
    _check("wsum", host(wsum2), host(wsum), dt)
