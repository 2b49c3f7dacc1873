"""GPU parity of the tcgen05 tensor-core backward (bf16, d = 32, G up to 4096,
padded inside the kernels to whole 128-slot blocks; past 640 slots every pass runs
over slot ranges) against the fp64 oracle, at both product arithmetics.

Each backward call runs in isolation, fed with the ORACLE's forward values
(mixed tokens, tokens, weight sums and lse), so that only the backward kernels
are checked:
  fs_deslice_bwd : d_tokens_mixed, dx_mid, dW, dbias, dtau
  fs_slice_bwd   : dx_mid, dfx, dW, dbias, dtau   (d_tokens drawn at random)
and the two calls chained with accumulate = 1 must add up.
Tolerance: relative L2 <= 1e-2 per tensor (bf16 inputs, fp32 accumulation).
"""
import numpy as np
import pytest
import torch

from oracle import flashslice_oracle as orc
from paper_2609_32525_gb300.workloads import make_case

from _parity import host, rel_l2, upload

pytestmark = pytest.mark.gpu

# (B, N, H, G): two points, exactly one tile, ragged tails, several heads and
# batches, every supported slot count class.
SHAPES = [
    (1, 2, 1, 128),
    (2, 7, 2, 256),
    (1, 33, 1, 384),
    (1, 128, 1, 128),
    (1, 129, 2, 256),
    (2, 1000, 3, 384),
    (1, 5000, 2, 512),
    (1, 3001, 1, 640),
    (2, 2049, 2, 256),
    (1, 1000, 2, 100),  # G padded to 128 inside the kernels
    (2, 777, 1, 48),
]
# G past 640: the passes run over 2, 2, 3 and 8 slot ranges (the last one ragged
# for G = 700 and 1500).
RANGED = [
    (1, 300, 2, 700),
    (1, 2000, 2, 1024),
    (2, 129, 1, 1500),
    (1, 257, 1, 4096),
]
TOL = 1e-2


def _f32(a, device="cuda"):
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(device)


def _run(lib, wl, dev, dot, accumulate=False, path=1):
    s = lib.shape_of(dev["x_mid"], wl.G, wl.eps, dot=dot)
    assert lib.backward_path_for_shape(s) == path
    fw = orc.forward(wl.x_mid, wl.fx, wl.W_slice, wl.bias, wl.tau, wl.M, eps=wl.eps,
                     points=np.array([], dtype=np.int64))
    ref_lse = fw["lse"].transpose(0, 2, 1)  # [B,H,N]
    B, N, H, G, d = wl.B, wl.N, wl.H, wl.G, wl.d
    rng = np.random.default_rng(1234 + N + G)
    d_tokens = rng.standard_normal((B, H, G, d))
    f32 = dict(dtype=torch.float32, device="cuda")
    out = {}
    dzm = torch.full((B, H, G, d), float("nan"), **f32)
    dx = torch.zeros(B, N, H, d, dtype=torch.bfloat16, device="cuda")
    dW = torch.zeros(H, d, G, **f32)
    db = torch.zeros(H, G, **f32)
    dt = torch.zeros(H, **f32)
    ws = lib.workspace(s, lib.FS_OP_DESLICE_BWD)
    lib.fs_deslice_bwd(s, dev["x_mid"], dev["W_slice"], dev["bias"], dev["tau"], _f32(fw["tokens_mixed"]),
                       _f32(ref_lse), dev["dout"], dzm, dx, dW, db, dt, False, ws)
    torch.cuda.synchronize()
    assert lib.fs_device_status(ws) == lib.FS_OK
    out["deslice"] = {"d_tokens_mixed": host(dzm), "dx_mid": host(dx), "dW": host(dW), "dbias": host(db),
                      "dtau": host(dt)}
    dx2 = dx.clone() if accumulate else torch.zeros_like(dx)
    dW2, db2, dt2 = (dW.clone(), db.clone(), dt.clone()) if accumulate else (
        torch.zeros_like(dW), torch.zeros_like(db), torch.zeros_like(dt))
    dfx = torch.full((B, N, H, d), float("nan"), dtype=torch.bfloat16, device="cuda")
    ws2 = lib.workspace(s, lib.FS_OP_SLICE_BWD)
    lib.fs_slice_bwd(s, dev["x_mid"], dev["fx"], dev["W_slice"], dev["bias"], dev["tau"], _f32(fw["tokens"]),
                     _f32(fw["wsum"]), _f32(ref_lse), _f32(d_tokens), dx2, dfx, dW2, db2, dt2, accumulate, ws2)
    torch.cuda.synchronize()
    assert lib.fs_device_status(ws2) == lib.FS_OK
    out["slice"] = {"dx_mid": host(dx2), "dfx": host(dfx), "dW": host(dW2), "dbias": host(db2), "dtau": host(dt2)}
    refs = {
        "deslice": orc.deslice_bwd(wl.x_mid, wl.W_slice, wl.bias, wl.tau, fw["tokens_mixed"], wl.dout),
        "slice": orc.slice_bwd(wl.x_mid, wl.fx, wl.W_slice, wl.bias, wl.tau, fw["tokens"], fw["wsum"], d_tokens,
                               eps=wl.eps),
    }
    return out, refs


@pytest.mark.parametrize("dot", ["bf16", "bf16x2"])
@pytest.mark.parametrize("shp", SHAPES + RANGED, ids=lambda s: "B{}N{}H{}G{}".format(*s))
def test_tc_backward_calls(lib, shp, dot):
    B, N, H, G = shp
    wl = make_case(B, N, H, 32, G, dtype="bf16", seed=600 + N + G, backward=True)
    dev = upload(wl)
    dotc = lib.FS_DOT_BF16X2 if dot == "bf16x2" else lib.FS_DOT_BF16
    got, ref = _run(lib, wl, dev, dotc)
    errs = {}
    for call in ("deslice", "slice"):
        for k, v in got[call].items():
            errs[f"{call}.{k}"] = rel_l2(v, ref[call][k])
    print(shp, dot, " ".join("{}={:.2e}".format(k, e) for k, e in errs.items()))
    bad = {k: e for k, e in errs.items() if not e <= TOL}
    assert not bad, "rel L2 above {:.0e}: {}".format(TOL, {k: "{:.3e}".format(e) for k, e in bad.items()})


@pytest.mark.parametrize("G", [256, 1024])
def test_tc_backward_accumulates(lib, G):
    wl = make_case(2, 1500, 2, 32, G, dtype="bf16", seed=611 + G, backward=True)
    dev = upload(wl)
    got, ref = _run(lib, wl, dev, lib.FS_DOT_BF16X2, accumulate=True)
    for k in ("dx_mid", "dW", "dbias", "dtau"):
        want = ref["deslice"][k] + ref["slice"][k]
        e = rel_l2(got["slice"][k], want)
        assert e <= TOL, f"{k}: {e:.3e}"


def test_single_point_takes_the_simt_backward(lib):
    """N = 1: every token is the point's fx times S/(S + eps), the slice gradients
    are O(eps); the fp32 SIMT backward resolves them."""
    wl = make_case(1, 1, 1, 32, 128, dtype="bf16", seed=601, backward=True)
    dev = upload(wl)
    got, ref = _run(lib, wl, dev, lib.FS_DOT_BF16X2, path=0)
    for call in ("deslice", "slice"):
        for k, v in got[call].items():
            e = rel_l2(v, ref[call][k])
            assert e <= TOL, f"{call}.{k}: {e:.3e}"


def test_backward_path_by_shape(lib):
    """bf16, d = 32: the tensor-core backward up to the header's G = 4096 (slot
    ranges past 640), the SIMT backward for other head widths."""
    assert lib.backward_path_for_shape(lib.make_shape(1, 4096, 2, 32, 1024, lib.FS_BF16)) == 1
    assert lib.backward_path_for_shape(lib.make_shape(1, 4096, 2, 32, 4096, lib.FS_BF16)) == 1
    assert lib.path_for_shape(lib.make_shape(1, 4096, 2, 32, 4096, lib.FS_BF16)) == 0
    assert lib.backward_path_for_shape(lib.make_shape(1, 4096, 2, 64, 1024, lib.FS_BF16)) == 0
