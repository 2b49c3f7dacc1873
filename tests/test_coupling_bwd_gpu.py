"""GPU parity of fs_coupling_bwd, the coupling's whole backward in one call,
against the fp64 oracle, and against the three separate calls (fs_deslice_bwd,
fs_mix_bwd, fs_slice_bwd).  On the tensor-core backward its single point pass
forms dx from the sum of both calls' da; it runs over slot ranges of at most 256
(G = 384 as three of 128, G = 512 as two of 256, G = 1024 as four of 256 beside
the other passes' two of 512), on shapes with one and with many point tiles per CTA.  Tolerances as in tests/_parity.py: bf16 inputs
relative L2 <= 1e-2, fp32 inputs normwise max relative <= 1e-4."""
import numpy as np
import pytest
import torch

from paper_2609_32525_gb300.workloads import make_case

from _parity import error, host, oracle_backward, tol, upload

pytestmark = pytest.mark.gpu

# (B, N, H, d, G, dtype, dot)
SHAPES = [
    (1, 2, 1, 32, 128, "bf16", "bf16x2"),
    (2, 1000, 2, 32, 100, "bf16", "bf16x2"),
    (1, 3001, 2, 32, 256, "bf16", "bf16"),
    (2, 777, 1, 32, 384, "bf16", "bf16x2"),
    (1, 2049, 2, 32, 512, "bf16", "bf16x2"),
    (1, 1500, 1, 32, 1024, "bf16", "bf16x2"),
    # many point tiles per CTA (the passes' pipelines wrap around their buffers)
    (1, 20000, 8, 32, 256, "bf16", "bf16x2"),
    (2, 9000, 4, 32, 512, "bf16", "bf16x2"),
    (1, 900, 2, 32, 48, "f32", "bf16"),
    (1, 500, 2, 16, 40, "bf16", "bf16"),
]
GRADS = ("dx_mid", "dfx", "dW", "dbias", "dtau", "dM")


def _ids(s):
    return "B{}N{}H{}d{}G{}-{}-{}".format(*s)


@pytest.mark.parametrize("shp", SHAPES, ids=_ids)
def test_coupling_bwd_against_the_oracle_and_the_separate_calls(lib, shp):
    B, N, H, d, G, dtype, dot = shp
    wl = make_case(B, N, H, d, G, dtype=dtype, seed=2100 + G + N, backward=True)
    dev = upload(wl)
    dotc = lib.FS_DOT_BF16X2 if dot == "bf16x2" else lib.FS_DOT_BF16
    c2 = lib.Coupling(B, N, H, d, G, torch.bfloat16 if dtype == "bf16" else torch.float32, wl.eps, backward=True,
                      dot=dotc)
    c2.forward(dev["x_mid"], dev["fx"], dev["W_slice"], dev["bias"], dev["tau"], dev["M"])
    args = (dev["x_mid"], dev["fx"], dev["W_slice"], dev["bias"], dev["tau"], dev["M"], dev["dout"])
    fused = {k: v.clone() for k, v in c2.backward(*args, fused=True).items()}
    fused["d_tokens_mixed"] = c2.d_tokens_mixed.clone()
    sep = c2.backward(*args, fused=False)
    torch.cuda.synchronize()
    assert c2.device_status() == lib.FS_OK
    rb = oracle_backward(wl)
    errs = {k: error(host(fused[k]), rb[k], dtype) for k in GRADS + ("d_tokens_mixed",)}
    print(_ids(shp), "path", lib.backward_path_for_shape(c2.shape),
          " ".join("{}={:.2e}".format(k, e) for k, e in errs.items()))
    bad = {k: e for k, e in errs.items() if not e <= tol(dtype)}
    assert not bad, {k: "{:.3e}".format(e) for k, e in bad.items()}
    # against the separate calls: the same sums up to rounding (the fused dx is rounded
    # to bf16 once, the separate calls' twice: ~2^-9 relative apart)
    for k in GRADS:
        e = error(host(fused[k]), host(sep[k]), dtype)
        assert e <= tol(dtype) / 2, f"{k}: fused against separate {e:.3e}"


def test_coupling_bwd_accumulates(lib):
    """accumulate = 1 adds the whole backward to dx_mid, dW, dbias, dtau."""
    wl = make_case(2, 1200, 2, 32, 512, dtype="bf16", seed=2200, backward=True)
    dev = upload(wl)
    c = lib.Coupling(wl.B, wl.N, wl.H, 32, wl.G, torch.bfloat16, wl.eps, backward=True)
    c.forward(dev["x_mid"], dev["fx"], dev["W_slice"], dev["bias"], dev["tau"], dev["M"])
    args = (dev["x_mid"], dev["fx"], dev["W_slice"], dev["bias"], dev["tau"], dev["M"], dev["dout"])
    once = {k: v.clone() for k, v in c.backward(*args).items()}
    s = c.shape
    lib.fs_coupling_bwd(s, dev["x_mid"], dev["fx"], dev["W_slice"], dev["bias"], dev["tau"], dev["M"], c.tokens,
                        c.wsum, c.tokens_mixed, c.lse, dev["dout"], c.d_tokens_mixed, c.d_tokens, c.dx_mid, c.dfx,
                        c.dW, c.dbias, c.dtau, c.dM, True, c.ws_cbwd)
    torch.cuda.synchronize()
    assert c.device_status() == lib.FS_OK
    for k in ("dx_mid", "dW", "dbias", "dtau"):
        e = error(host(getattr(c, k)), 2 * host(once[k]), "bf16")
        assert e <= 1e-2, f"{k}: {e:.3e}"
    np.testing.assert_array_equal(host(c.dM), host(once["dM"]))
