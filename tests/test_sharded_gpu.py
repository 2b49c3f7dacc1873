"""The point-sharded coupling (App. G.4) through the C ABI on one GPU: the ranks'
shards run one after another, and their partials are summed in a fixed order
(shard 0 first) where the ranks would all-reduce them.

Forward per shard: fs_slice_fwd(finalize = 0) gives its unnormalised U and S; the
summed U, S go through fs_slice_finalize and fs_mix; each shard deslices its own
points with its own lse.  Backward per shard: fs_deslice_bwd gives its partial
d_tokens_mixed; the sum goes through fs_mix_bwd; fs_slice_bwd runs on the shard's
points with the global tokens and weight sums; dW, dbias, dtau are summed over
the shards.  Every result is compared with the unsharded fp64 oracle at the
usual bars (fp32 normwise max relative 1e-4, bf16 relative L2 1e-2), and with
the unsharded GPU calls.
"""
import numpy as np
import pytest
import torch

from oracle import flashslice_oracle as orc
from paper_2609_32525_gb300 import sharding
from paper_2609_32525_gb300.workloads import make_case

from _parity import error, host, tol, upload

pytestmark = pytest.mark.gpu

# tensor-core bf16 (d = 32; G = 256 and a padded G = 100), SIMT fp32 (d = 16)
CASES = [(2, 3001, 2, 32, 256, "bf16", 3), (1, 2500, 2, 32, 100, "bf16", 2), (2, 1201, 2, 16, 40, "f32", 3)]
IDS = ["tc-G256-3shards", "tc-G100-2shards", "simt-f32-3shards"]


def _buffers(lib, s, x):
    """One shard's (or the whole problem's) outputs and workspaces."""
    B, N, H, d = x.shape
    G = s.G
    f32 = dict(dtype=torch.float32, device="cuda")
    o = {"U": torch.empty(B, H, G, d, **f32), "S": torch.empty(B, H, G, **f32), "lse": torch.empty(B, H, N, **f32),
         "out": torch.empty_like(x), "dzm": torch.empty(B, H, G, d, **f32), "dx": torch.empty_like(x),
         "dfx": torch.empty_like(x), "dW": torch.empty(H, d, G, **f32), "db": torch.empty(H, G, **f32),
         "dt": torch.empty(H, **f32)}
    o["ws"] = {op: lib.workspace(s, op) for op in (lib.FS_OP_SLICE_FWD, lib.FS_OP_DESLICE_FWD,
                                                   lib.FS_OP_DESLICE_BWD, lib.FS_OP_SLICE_BWD)}
    return o


def _run(lib, dev, G, eps, shards):
    """The sharded coupling forward and backward; shards = [(n0, n1)]."""
    args = (dev["W_slice"], dev["bias"], dev["tau"])
    parts = []
    for n0, n1 in shards:
        x = dev["x_mid"][:, n0:n1].contiguous()
        f = dev["fx"][:, n0:n1].contiguous()
        do = dev["dout"][:, n0:n1].contiguous()
        s = lib.shape_of(x, G, eps, dot=lib.FS_DOT_BF16X2)
        o = _buffers(lib, s, x)
        o.update(x=x, f=f, do=do, s=s)
        lib.fs_slice_fwd(s, x, f, *args, o["U"], o["S"], o["lse"], False, o["ws"][lib.FS_OP_SLICE_FWD])
        parts.append(o)
    # the forward exchange: sums of the unnormalised partials, shard 0 first
    U, S = parts[0]["U"].clone(), parts[0]["S"].clone()
    for o in parts[1:]:
        U += o["U"]
        S += o["S"]
    s0 = parts[0]["s"]
    tokens = U.clone()
    lib.fs_slice_finalize(s0, tokens, S)
    tm = torch.empty_like(tokens)
    lib.fs_mix(s0, dev["M"], tokens, tm)
    for o in parts:
        lib.fs_deslice_fwd(o["s"], o["x"], *args, tm, o["lse"], o["out"], o["ws"][lib.FS_OP_DESLICE_FWD])
        lib.fs_deslice_bwd(o["s"], o["x"], *args, tm, o["lse"], o["do"], o["dzm"], o["dx"], o["dW"], o["db"],
                           o["dt"], False, o["ws"][lib.FS_OP_DESLICE_BWD])
    # the backward exchange: the partial d_tokens_mixed
    dzm = parts[0]["dzm"].clone()
    for o in parts[1:]:
        dzm += o["dzm"]
    dz = torch.empty_like(dzm)
    dM = torch.empty(dev["M"].shape, dtype=torch.float32, device="cuda")
    lib.fs_mix_bwd(s0, dev["M"], tokens, dzm, dz, dM)
    for o in parts:
        lib.fs_slice_bwd(o["s"], o["x"], o["f"], *args, tokens, S, o["lse"], dz, o["dx"], o["dfx"], o["dW"], o["db"],
                         o["dt"], True, o["ws"][lib.FS_OP_SLICE_BWD])
    torch.cuda.synchronize()
    for o in parts:
        for w in o["ws"].values():
            assert lib.fs_device_status(w) == lib.FS_OK
    # the parameter gradients: summed over the shards, shard 0 first
    grads = {k: parts[0][k].clone() for k in ("dW", "db", "dt")}
    for o in parts[1:]:
        for k in grads:
            grads[k] += o[k]
    cat = lambda k: torch.cat([o[k] for o in parts], dim=1)  # noqa: E731
    return {"tokens": tokens, "wsum": S, "tokens_mixed": tm, "out": cat("out"), "d_tokens_mixed": dzm, "dM": dM,
            "dx_mid": cat("dx"), "dfx": cat("dfx"), "dW": grads["dW"], "dbias": grads["db"], "dtau": grads["dt"]}


@pytest.mark.parametrize("case", CASES, ids=IDS)
def test_point_shards_match_the_unsharded_coupling(lib, case):
    B, N, H, d, G, dt, R = case
    wl = make_case(B, N, H, d, G, dtype=dt, seed=1100 + G + R, backward=True)
    dev = upload(wl)
    shards = [sharding.point_range(N, r, R) for r in range(R)]
    got = _run(lib, dev, G, wl.eps, shards)
    whole = _run(lib, dev, G, wl.eps, [(0, N)])

    ref = orc.forward(wl.x_mid, wl.fx, wl.W_slice, wl.bias, wl.tau, wl.M, eps=wl.eps)
    rb = orc.backward(wl.x_mid, wl.fx, wl.W_slice, wl.bias, wl.tau, wl.M, wl.dout, eps=wl.eps)
    rd = orc.deslice_bwd(wl.x_mid, wl.W_slice, wl.bias, wl.tau, ref["tokens_mixed"], wl.dout)
    refs = {"tokens": ref["tokens"], "wsum": ref["wsum"], "tokens_mixed": ref["tokens_mixed"], "out": ref["out"],
            "d_tokens_mixed": rd["d_tokens_mixed"], "dM": rb["dM"], "dx_mid": rb["dx_mid"], "dfx": rb["dfx"],
            "dW": rb["dW"], "dbias": rb["dbias"], "dtau": rb["dtau"]}
    bad = {}
    for k, r in refs.items():
        e = error(host(got[k]), r, dt)
        e_whole = error(host(got[k]), host(whole[k]), dt)
        if not (e <= tol(dt) and e_whole <= tol(dt)):
            bad[k] = "vs oracle {:.2e}, vs unsharded GPU {:.2e}".format(e, e_whole)
    assert not bad, bad
