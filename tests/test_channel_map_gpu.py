"""GPU parity of the attention-free core (NoTokenAttn: a per-token channel map,
Sec. 2 after Eq. (1)) against the fp64 oracle.

* fs_mix_channels and fs_mix_channels_bwd alone, fp32 tokens, d = 16, 32, 64:
  normwise max relative error <= 1e-4 (fp32 arithmetic).
* A whole NoTokenAttn coupling through the C ABI on the tensor-core path (bf16):
  slice -> channel map -> deslice, then deslice backward -> channel-map backward ->
  slice backward; every output and gradient within relative L2 1e-2.
"""
import numpy as np
import pytest
import torch

from oracle import flashslice_oracle as orc
from paper_2609_32525_gb300.workloads import make_case

from _parity import error, host, max_rel, tol, upload

pytestmark = pytest.mark.gpu


def _f32(a):
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).cuda()


@pytest.mark.parametrize("shp", [(1, 2, 32, 16), (2, 8, 100, 32), (1, 3, 7, 64)], ids=lambda s: "B{}H{}G{}d{}".format(*s))
def test_channel_map_calls(lib, shp):
    B, H, G, d = shp
    rng = np.random.default_rng(70 + G)
    Wc, z, dzp = (rng.standard_normal((H, d, d)).astype(np.float32), rng.standard_normal((B, H, G, d)).astype(np.float32),
                  rng.standard_normal((B, H, G, d)).astype(np.float32))
    s = lib.make_shape(B, 16, H, d, G, lib.FS_F32)
    out, dz, dWc = torch.empty(B, H, G, d).cuda(), torch.empty(B, H, G, d).cuda(), torch.empty(H, d, d).cuda()
    lib.fs_mix_channels(s, _f32(Wc), _f32(z), out)
    lib.fs_mix_channels_bwd(s, _f32(Wc), _f32(z), _f32(dzp), dz, dWc)
    torch.cuda.synchronize()
    bw = orc.mix_channels_bwd(Wc, z, dzp)
    for name, got, ref in (("tokens_mixed", out, orc.mix_channels(Wc, z)), ("d_tokens", dz, bw["d_tokens"]),
                           ("dWc", dWc, bw["dWc"])):
        e = max_rel(host(got), ref)
        assert e <= 1e-4, f"{name}: {e:.3e}"


def test_notokenattn_coupling_forward_and_backward(lib):
    B, N, H, d, G = 2, 2000, 2, 32, 256
    wl = make_case(B, N, H, d, G, dtype="bf16", seed=71, backward=True)
    dev = upload(wl)
    Wc = np.eye(d)[None].repeat(H, 0) + 0.1 * np.random.default_rng(72).standard_normal((H, d, d))
    Wcd = _f32(Wc)
    s = lib.shape_of(dev["x_mid"], G, wl.eps, dot=lib.FS_DOT_BF16X2)
    f32 = dict(dtype=torch.float32, device="cuda")
    bf = dict(dtype=torch.bfloat16, device="cuda")
    tokens, wsum, lse = torch.empty(B, H, G, d, **f32), torch.empty(B, H, G, **f32), torch.empty(B, H, N, **f32)
    tm, out = torch.empty(B, H, G, d, **f32), torch.empty(B, N, H, d, **bf)
    ws = {op: lib.workspace(s, op) for op in (lib.FS_OP_SLICE_FWD, lib.FS_OP_DESLICE_FWD, lib.FS_OP_DESLICE_BWD,
                                               lib.FS_OP_SLICE_BWD)}
    args = (dev["W_slice"], dev["bias"], dev["tau"])
    lib.fs_slice_fwd(s, dev["x_mid"], dev["fx"], *args, tokens, wsum, lse, True, ws[lib.FS_OP_SLICE_FWD])
    lib.fs_mix_channels(s, Wcd, tokens, tm)
    lib.fs_deslice_fwd(s, dev["x_mid"], *args, tm, lse, out, ws[lib.FS_OP_DESLICE_FWD])
    dzm, dz, dWc = torch.empty(B, H, G, d, **f32), torch.empty(B, H, G, d, **f32), torch.empty(H, d, d, **f32)
    dx, dfx = torch.empty(B, N, H, d, **bf), torch.empty(B, N, H, d, **bf)
    dW, db, dt = torch.empty(H, d, G, **f32), torch.empty(H, G, **f32), torch.empty(H, **f32)
    lib.fs_deslice_bwd(s, dev["x_mid"], *args, tm, lse, dev["dout"], dzm, dx, dW, db, dt, False,
                       ws[lib.FS_OP_DESLICE_BWD])
    lib.fs_mix_channels_bwd(s, Wcd, tokens, dzm, dz, dWc)
    lib.fs_slice_bwd(s, dev["x_mid"], dev["fx"], *args, tokens, wsum, lse, dz, dx, dfx, dW, db, dt, True,
                     ws[lib.FS_OP_SLICE_BWD])
    torch.cuda.synchronize()
    for w in ws.values():
        assert lib.fs_device_status(w) == lib.FS_OK

    rs = orc.slice_fwd(wl.x_mid, wl.fx, wl.W_slice, wl.bias, wl.tau, eps=wl.eps)
    rtm = orc.mix_channels(Wc, rs["tokens"])
    rout = orc.deslice_fwd(wl.x_mid, wl.W_slice, wl.bias, wl.tau, rtm)
    rd = orc.deslice_bwd(wl.x_mid, wl.W_slice, wl.bias, wl.tau, rtm, wl.dout)
    rc = orc.mix_channels_bwd(Wc, rs["tokens"], rd["d_tokens_mixed"])
    rb = orc.slice_bwd(wl.x_mid, wl.fx, wl.W_slice, wl.bias, wl.tau, rs["tokens"], rs["wsum"], rc["d_tokens"],
                       eps=wl.eps)
    checks = (("out", out, rout), ("tokens_mixed", tm, rtm), ("d_tokens_mixed", dzm, rd["d_tokens_mixed"]),
              ("dWc", dWc, rc["dWc"]), ("dx_mid", dx, rd["dx_mid"] + rb["dx_mid"]), ("dfx", dfx, rb["dfx"]),
              ("dW", dW, rd["dW"] + rb["dW"]), ("dbias", db, rd["dbias"] + rb["dbias"]),
              ("dtau", dt, rd["dtau"] + rb["dtau"]))
    for name, got, ref in checks:
        e = error(host(got), ref, "bf16")
        assert e <= tol("bf16"), f"{name}: {e:.3e}"
