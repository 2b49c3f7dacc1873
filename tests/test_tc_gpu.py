"""GPU parity of the tcgen05 tensor-core forward kernels (bf16 inputs, G a
multiple of 128) against the fp64 oracle, each kernel checked in isolation:

  statistics : lse from fs_slice_fwd vs the oracle's log-sum-exp
  slice      : tokens / weight sums from fs_slice_fwd
  deslice    : fs_deslice_fwd fed with the ORACLE's lse and mixed tokens

Both product arithmetics are checked (FS_DOT_BF16 and the split FS_DOT_BF16X2).
Tolerance: relative L2 <= 1e-2 per tensor (bf16 inputs, fp32 accumulation),
1e-3 for tokens and weight sums with split products; lse is compared in
absolute nats against a bound derived from each arithmetic.
"""
import numpy as np
import pytest
import torch

from oracle import flashslice_oracle as orc
from paper_2609_32525_gb300.workloads import make_case

from _parity import host, rel_l2, upload

pytestmark = pytest.mark.gpu

# (B, N, H, G): ragged tails (N % 128 != 0), a single point, exactly one tile,
# one slice range (G <= 512) and two (G = 1024), several heads and batches.
SHAPES = [
    (1, 1, 1, 128),
    (1, 128, 1, 128),
    (1, 129, 2, 256),
    (2, 1000, 3, 384),
    (1, 5000, 2, 512),
    (1, 3001, 1, 640),
    (1, 4000, 2, 1024),
    (2, 2049, 8, 256),
]


def _lse_bhn(ref):
    return ref["lse"].transpose(0, 2, 1)


def lse_error_bound(wl, split):
    """Per-point bound on |lse_gpu - lse_exact| [B,H,N] implied by the arithmetic:
    the statistics pass forms the logits with W' = W log2(e)/tau rounded to
    bf16 (relative error <= 2^-8), or with split products as two bf16 halves,
    hi + lo (residual <= 2^-16); x is bf16 already, exact; the bias rides as two
    halves (<= 2^-16); accumulation is fp32.  lse is a smooth maximum of the
    logits, so its error is at most the largest logit error of the point."""
    B, N, H, d, G = wl.B, wl.N, wl.H, wl.d, wl.G
    out = np.empty((B, H, N))
    for h in range(H):
        Wp = np.abs(wl.W_slice[h].astype(np.float64)) * np.log2(np.e) / wl.tau[h]
        bp = np.abs(wl.bias[h].astype(np.float64)).max() * np.log2(np.e) / wl.tau[h]
        for b in range(B):
            s = np.abs(wl.x_mid[b, :, h, :].astype(np.float64)) @ Wp  # N x G
            rel = 2.0 ** -16 if split else 2.0 ** -8
            out[b, h] = np.log(2.0) * (rel * s.max(axis=1) + 2.0 ** -16 * bp) + 1e-4
    return out


@pytest.mark.parametrize("dot", ["bf16", "bf16x2"])
@pytest.mark.parametrize("shp", SHAPES, ids=lambda s: "B{}N{}H{}G{}".format(*s))
def test_tc_forward_kernels(lib, shp, dot):
    B, N, H, G = shp
    wl = make_case(B, N, H, 32, G, dtype="bf16", seed=300 + N + G, backward=False)
    dev = upload(wl)
    split = dot == "bf16x2"
    s = lib.shape_of(dev["x_mid"], G, wl.eps, lib.FS_DOT_BF16X2 if split else lib.FS_DOT_BF16)
    assert lib.path_for_shape(s) == 1, "shape should take the tensor-core path"
    ref = orc.forward(wl.x_mid, wl.fx, wl.W_slice, wl.bias, wl.tau, wl.M, eps=wl.eps)

    f32 = dict(dtype=torch.float32, device="cuda")
    tokens = torch.empty(B, H, G, 32, **f32)
    wsum = torch.empty(B, H, G, **f32)
    lse = torch.empty(B, H, N, **f32)
    ws = lib.workspace(s, lib.FS_OP_SLICE_FWD)
    lib.fs_slice_fwd(s, dev["x_mid"], dev["fx"], dev["W_slice"], dev["bias"], dev["tau"], tokens, wsum, lse, True, ws)
    torch.cuda.synchronize()
    assert lib.fs_device_status(ws) == lib.FS_OK
    lse_dev = np.abs(host(lse) - _lse_bhn(ref))
    bound = lse_error_bound(wl, split)
    worst = (lse_dev / bound).max()
    assert worst <= 1.0, f"lse error exceeds its bound: max ratio {worst:.3f}, max abs {lse_dev.max():.3e}"
    e_tok = rel_l2(host(tokens), ref["tokens"])
    e_ws = rel_l2(host(wsum), ref["wsum"])
    # Split products carry the weights and W' to ~2^-16: tokens and weight sums
    # to ~1e-4 (checked at 1e-3); bf16 products to the contract's 1e-2.
    t_tol = 1e-3 if split else 1e-2
    assert e_ws < t_tol, f"wsum rel L2 {e_ws:.3e}"
    assert e_tok < t_tol, f"tokens rel L2 {e_tok:.3e}"

    # Deslice in isolation: the oracle's statistics and mixed tokens as inputs.
    ref_lse = torch.from_numpy(np.ascontiguousarray(_lse_bhn(ref)).astype(np.float32)).cuda()
    ref_tm = torch.from_numpy(ref["tokens_mixed"].astype(np.float32)).cuda()
    out = torch.empty_like(dev["x_mid"])
    wsd = lib.workspace(s, lib.FS_OP_DESLICE_FWD)
    lib.fs_deslice_fwd(s, dev["x_mid"], dev["W_slice"], dev["bias"], dev["tau"], ref_tm, ref_lse, out, wsd)
    torch.cuda.synchronize()
    assert lib.fs_device_status(wsd) == lib.FS_OK
    e_out = rel_l2(host(out), ref["out"])
    assert e_out < 1e-2, f"deslice out rel L2 {e_out:.3e}"

    # Deslice without statistics (computes them itself).
    out2 = torch.empty_like(dev["x_mid"])
    lib.fs_deslice_fwd(s, dev["x_mid"], dev["W_slice"], dev["bias"], dev["tau"], ref_tm, None, out2, wsd)
    torch.cuda.synchronize()
    e_out2 = rel_l2(host(out2), ref["out"])
    assert e_out2 < 1e-2, f"deslice (own stats) out rel L2 {e_out2:.3e}"


def test_tc_full_chain_and_determinism(lib):
    wl = make_case(2, 3000, 4, 32, 512, dtype="bf16", seed=77, backward=False)
    dev = upload(wl)
    ref = orc.forward(wl.x_mid, wl.fx, wl.W_slice, wl.bias, wl.tau, wl.M, eps=wl.eps)
    outs = []
    for _ in range(2):
        c = lib.Coupling(wl.B, wl.N, wl.H, wl.d, wl.G, torch.bfloat16, wl.eps)
        c.forward(dev["x_mid"], dev["fx"], dev["W_slice"], dev["bias"], dev["tau"], dev["M"])
        torch.cuda.synchronize()
        assert c.device_status() == lib.FS_OK
        outs.append((c.out.clone(), c.tokens.clone()))
    assert rel_l2(host(outs[0][0]), ref["out"]) < 1e-2
    assert torch.equal(outs[0][0].view(torch.int16), outs[1][0].view(torch.int16))
    assert torch.equal(outs[0][1].view(torch.int32), outs[1][1].view(torch.int32))


@pytest.mark.parametrize("dot", ["bf16", "bf16x2"])
def test_tc_forward_then_backward(lib, dot):
    """The backward after a tensor-core forward, at both product arithmetics: with
    bf16 products the backward recomputes lse with split products; with split
    products it takes the forward's.  Every gradient against the oracle."""
    wl = make_case(2, 3000, 2, 32, 256, dtype="bf16", seed=88, backward=True)
    dev = upload(wl)
    c = lib.Coupling(wl.B, wl.N, wl.H, wl.d, wl.G, torch.bfloat16, wl.eps, backward=True,
                     dot=lib.FS_DOT_BF16X2 if dot == "bf16x2" else lib.FS_DOT_BF16)
    assert lib.path_for_shape(c.shape) == 1
    c.forward(dev["x_mid"], dev["fx"], dev["W_slice"], dev["bias"], dev["tau"], dev["M"])
    g = c.backward(dev["x_mid"], dev["fx"], dev["W_slice"], dev["bias"], dev["tau"], dev["M"], dev["dout"])
    torch.cuda.synchronize()
    assert c.device_status() == lib.FS_OK
    ref = orc.backward(wl.x_mid, wl.fx, wl.W_slice, wl.bias, wl.tau, wl.M, wl.dout, eps=wl.eps)
    for k in ("dx_mid", "dfx", "dW", "dbias", "dtau", "dM"):
        e = rel_l2(host(g[k]), ref[k])
        assert e < 1e-2, f"{k} rel L2 {e:.3e}"
