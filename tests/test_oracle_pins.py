"""Pins for the fp64 CPU oracle: values fixed by the paper's definitions and by
mathematics, chosen so that a plausible slip in the oracle (a dropped term, a
wrong sign, a transposed operand, a misplaced temperature or epsilon) fails at
least one of them.  No GPU involved.
"""
import json
import math
import os
from fractions import Fraction

import numpy as np
import pytest

from oracle import bruteforce
from oracle import flashslice_oracle as orc
from paper_2609_32525_gb300.workloads import make_case

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "worked_example.json")
LN2, LN3 = math.log(2.0), math.log(3.0)


def _q(s):
    return float(Fraction(s))


def _worked_inputs():
    x = np.array([2 * LN3, 0.0]).reshape(1, 2, 1, 1)
    fx = np.array([4.0, 8.0]).reshape(1, 2, 1, 1)
    W = np.array([[[1.0, 0.0]]])
    bias = np.array([[0.0, 2 * LN2]])
    tau = np.array([2.0])
    M = np.array([[[1.0, 1.0], [0.0, 1.0]]])
    dout = np.array([1.0, 0.0]).reshape(1, 2, 1, 1)
    return x, fx, W, bias, tau, M, dout


def test_worked_example_forward():
    """Hand-derived values (tests/golden/worked_example.md) of Sec. 2 / Eq. (1)."""
    g = json.load(open(GOLDEN))["forward"]
    x, fx, W, bias, tau, M, _ = _worked_inputs()
    fw = orc.forward(x, fx, W, bias, tau, M, eps=0.0)
    np.testing.assert_allclose(fw["wsum"][0, 0], [_q(v) for v in g["wsum"]], rtol=1e-14)
    np.testing.assert_allclose(fw["tokens"][0, 0, :, 0], [_q(v) for v in g["tokens"]], rtol=1e-14)
    np.testing.assert_allclose(fw["tokens_mixed"][0, 0, :, 0], [_q(v) for v in g["tokens_mixed"]], rtol=1e-14)
    np.testing.assert_allclose(fw["out"][0, :, 0, 0], [_q(v) for v in g["out"]], rtol=1e-14)
    np.testing.assert_allclose(fw["lse"][0, :, 0], [math.log(5.0), math.log(3.0)], rtol=1e-14)
    s = orc.slice_fwd(x, fx, W, bias, tau, eps=0.0, finalize=False)
    np.testing.assert_allclose(s["tokens"][0, 0, :, 0], [_q(v) for v in g["numerators"]], rtol=1e-14)
    a = orc.logits(x[0, :, 0, :], W[0], bias[0], tau[0])
    w, _ = orc.softmax_rows(a)
    np.testing.assert_allclose(w, [[_q(v) for v in r] for r in g["w"]], rtol=1e-14)


def test_worked_example_backward():
    g = json.load(open(GOLDEN))["backward"]
    x, fx, W, bias, tau, M, dout = _worked_inputs()
    bw = orc.backward(x, fx, W, bias, tau, M, dout, eps=0.0)
    np.testing.assert_allclose(bw["d_tokens_mixed"][0, 0, :, 0], [_q(v) for v in g["d_tokens_mixed"]], rtol=1e-14)
    np.testing.assert_allclose(bw["dM"][0], [[_q(v) for v in r] for r in g["dM"]], rtol=1e-14)
    np.testing.assert_allclose(bw["d_tokens"][0, 0, :, 0], [_q(v) for v in g["d_tokens"]], rtol=1e-14)
    np.testing.assert_allclose(bw["dfx"][0, :, 0, 0], [_q(v) for v in g["dfx"]], rtol=1e-14)
    np.testing.assert_allclose(bw["dbias"][0], [_q(v) for v in g["dbias"]], rtol=1e-13)
    np.testing.assert_allclose(bw["dx_mid"][0, :, 0, 0], [_q(v) for v in g["dx_mid"]], rtol=1e-13)
    c = 32241 / 19600
    np.testing.assert_allclose(bw["dW"][0, 0], [LN3 * c, -LN3 * c], rtol=1e-13)
    dtau = -0.5 * (c * math.log(1.5) - 43 / 784 * LN2)
    np.testing.assert_allclose(bw["dtau"][0], dtau, rtol=1e-12)


def _case_arrays(wl):
    return (wl.x_mid.astype(np.float64), wl.fx.astype(np.float64), wl.W_slice.astype(np.float64),
            wl.bias.astype(np.float64), wl.tau.astype(np.float64), wl.M.astype(np.float64),
            wl.dout.astype(np.float64))


TINY = dict(B=2, N=7, H=2, d=3, G=5)


def test_bruteforce_matches_oracle():
    """Scalar loops (no numpy contractions) vs the matrix formulation."""
    wl = make_case(**TINY, seed=11, bias_std=0.3)
    x, fx, W, b, t, M, dO = _case_arrays(wl)
    fw = orc.forward(x, fx, W, b, t, M, eps=wl.eps)
    bw = orc.backward(x, fx, W, b, t, M, dO, eps=wl.eps)
    args = (x.tolist(), fx.tolist(), W.tolist(), b.tolist(), t.tolist(), M.tolist(), wl.eps)
    tok, ws, tm, out = bruteforce.forward(*args, **{k: TINY[k] for k in "BNHdG"})
    np.testing.assert_allclose(np.array(tok), fw["tokens"], rtol=1e-12, atol=1e-13)
    np.testing.assert_allclose(np.array(ws), fw["wsum"], rtol=1e-12)
    np.testing.assert_allclose(np.array(tm), fw["tokens_mixed"], rtol=1e-12, atol=1e-13)
    np.testing.assert_allclose(np.array(out), fw["out"], rtol=1e-12, atol=1e-13)
    gb = bruteforce.backward(*args, dO.tolist(), **{k: TINY[k] for k in "BNHdG"})
    for key in ("dx_mid", "dfx", "dW", "dbias", "dtau", "dM"):
        np.testing.assert_allclose(np.array(gb[key]), bw[key], rtol=1e-11, atol=1e-12, err_msg=key)


def _loss(x, fx, W, b, t, M, dO, eps):
    return float((orc.forward(x, fx, W, b, t, M, eps=eps)["out"] * dO).sum())


def test_finite_differences_all_gradients():
    """Central differences in fp64 for every gradient (x_mid, fx, W, bias, tau, M)."""
    wl = make_case(**TINY, seed=5, bias_std=0.5)
    x, fx, W, b, t, M, dO = _case_arrays(wl)
    bw = orc.backward(x, fx, W, b, t, M, dO, eps=wl.eps)
    params = {"dx_mid": x, "dfx": fx, "dW": W, "dbias": b, "dtau": t, "dM": M}
    order = ["dx_mid", "dfx", "dW", "dbias", "dtau", "dM"]
    h = 1e-6
    for key in order:
        p = params[key]
        fd = np.zeros_like(p)
        for i in np.ndindex(p.shape):
            old = p[i]
            p[i] = old + h
            lp = _loss(x, fx, W, b, t, M, dO, wl.eps)
            p[i] = old - h
            lm = _loss(x, fx, W, b, t, M, dO, wl.eps)
            p[i] = old
            fd[i] = (lp - lm) / (2 * h)
        err = np.linalg.norm(fd - bw[key]) / np.linalg.norm(bw[key])
        assert err < 1e-6, (key, err)


def test_softmax_rows_partition_of_unity():
    wl = make_case(B=1, N=300, H=2, d=16, G=37, seed=3, bias_std=1.0)
    for h in range(2):
        a = orc.logits(wl.x_mid[0, :, h, :], wl.W_slice[h], wl.bias[h], wl.tau[h])
        w, lse = orc.softmax_rows(a)
        assert np.all(w >= 0)
        np.testing.assert_allclose(w.sum(axis=1), 1.0, atol=1e-14)
        np.testing.assert_allclose(np.exp(a - lse[:, None]), w, rtol=1e-12)


@pytest.mark.parametrize("mode", ["zero_logits", "huge_tau"])
def test_uniform_weights_give_global_mean(mode):
    """W = 0, beta = 0 (Prop. 1's construction) or tau -> inf: w = 1/G, every token
    equals sum_n f_n / (N + G eps)."""
    wl = make_case(B=2, N=50, H=3, d=4, G=6, seed=8, backward=False)
    W, b, t = wl.W_slice.astype(np.float64), wl.bias.astype(np.float64), wl.tau.astype(np.float64)
    if mode == "zero_logits":
        W[:] = 0.0
        b[:] = 0.0
    else:
        t[:] = 1e12
    fw = orc.forward(wl.x_mid, wl.fx, W, b, t, wl.M, eps=wl.eps)
    N, G = wl.N, wl.G
    for bb in range(2):
        for h in range(3):
            mean = wl.fx[bb, :, h, :].astype(np.float64).sum(axis=0) / (N + G * wl.eps)
            np.testing.assert_allclose(fw["tokens"][bb, h], np.broadcast_to(mean, (G, 4)), rtol=1e-9)
            np.testing.assert_allclose(fw["wsum"][bb, h], N / G, rtol=1e-9)


def test_single_slice_is_weighted_mean():
    """G = 1: w = 1, z = sum f / (N + eps), out_n = M z for every point."""
    wl = make_case(B=1, N=40, H=2, d=5, G=1, seed=9, backward=False)
    fw = orc.forward(wl.x_mid, wl.fx, wl.W_slice, wl.bias, wl.tau, wl.M, eps=wl.eps)
    for h in range(2):
        z = wl.fx[0, :, h, :].astype(np.float64).sum(axis=0) / (wl.N + wl.eps)
        np.testing.assert_allclose(fw["tokens"][0, h, 0], z, rtol=1e-12)
        np.testing.assert_allclose(fw["out"][0, :, h, :], np.broadcast_to(float(wl.M[h, 0, 0]) * z, (wl.N, 5)),
                                   rtol=1e-12)


def test_one_hot_limit_is_group_by():
    """tau -> 0: each point belongs to its argmax slot only; tokens are group means
    (count + eps denominator) and out_n = z'_{argmax n}."""
    wl = make_case(B=1, N=200, H=2, d=3, G=7, seed=10, backward=False)
    t = np.full(2, 1e-7)
    fw = orc.forward(wl.x_mid, wl.fx, wl.W_slice, wl.bias, t, wl.M, eps=wl.eps)
    for h in range(2):
        raw = wl.x_mid[0, :, h, :].astype(np.float64) @ wl.W_slice[h].astype(np.float64) + wl.bias[h]
        arg = raw.argmax(axis=1)
        z = np.zeros((7, 3))
        for g in range(7):
            sel = arg == g
            z[g] = wl.fx[0, sel, h, :].astype(np.float64).sum(axis=0) / (sel.sum() + wl.eps)
        np.testing.assert_allclose(fw["tokens"][0, h], z, rtol=1e-12, atol=1e-12)
        zp = wl.M[h].astype(np.float64) @ z
        np.testing.assert_allclose(fw["out"][0, :, h, :], zp[arg], rtol=1e-12, atol=1e-12)


def test_tokens_are_convex_combinations():
    wl = make_case(B=1, N=500, H=2, d=6, G=9, seed=12, backward=False)
    s = orc.slice_fwd(wl.x_mid, wl.fx, wl.W_slice, wl.bias, wl.tau, eps=0.0)
    for h in range(2):
        f = wl.fx[0, :, h, :]
        assert np.all(s["tokens"][0, h] <= f.max(axis=0) + 1e-12)
        assert np.all(s["tokens"][0, h] >= f.min(axis=0) - 1e-12)


def test_partition_of_unity_reproduces_constants():
    """M = I and fx = c with eps = 0: every token is c and out_n = c (sum_g w = 1)."""
    wl = make_case(B=1, N=64, H=2, d=4, G=8, seed=13, backward=False)
    fx = np.full_like(wl.fx, 0.0) + np.array([1.5, -2.0, 0.25, 3.0], np.float32)
    M = np.broadcast_to(np.eye(8), (2, 8, 8)).copy()
    fw = orc.forward(wl.x_mid, fx, wl.W_slice, wl.bias, wl.tau, M, eps=0.0)
    np.testing.assert_allclose(fw["out"], np.broadcast_to(fx, fw["out"].shape), rtol=1e-12)


def test_permuting_points():
    """Permuting the points leaves the tokens unchanged and permutes out."""
    wl = make_case(B=1, N=123, H=2, d=4, G=6, seed=14, backward=False)
    perm = np.random.default_rng(0).permutation(wl.N)
    f1 = orc.forward(wl.x_mid, wl.fx, wl.W_slice, wl.bias, wl.tau, wl.M, eps=wl.eps)
    f2 = orc.forward(wl.x_mid[:, perm], wl.fx[:, perm], wl.W_slice, wl.bias, wl.tau, wl.M, eps=wl.eps)
    np.testing.assert_allclose(f2["tokens"], f1["tokens"], rtol=1e-12)
    np.testing.assert_allclose(f2["out"], f1["out"][:, perm], rtol=1e-12)


def _grads(seed, **kw):
    wl = make_case(B=2, N=33, H=3, d=4, G=6, seed=seed, bias_std=0.4, **kw)
    x, fx, W, b, t, M, dO = _case_arrays(wl)
    fw = orc.forward(x, fx, W, b, t, M, eps=wl.eps)
    bw = orc.backward(x, fx, W, b, t, M, dO, eps=wl.eps)
    return wl, (x, fx, W, b, t, M, dO), fw, bw


def test_linearity_identities():
    """out is linear in fx and in M: <fx, dfx> = <out, dO> = <M, dM>."""
    _, (x, fx, W, b, t, M, dO), fw, bw = _grads(15)
    L = (fw["out"] * dO).sum()
    np.testing.assert_allclose((fx * bw["dfx"]).sum(), L, rtol=1e-12)
    np.testing.assert_allclose((M * bw["dM"]).sum(), L, rtol=1e-12)


def test_scale_invariance_pins_dtau():
    """(W_h, beta_h, tau_h) -> c(W_h, beta_h, tau_h) and (x_h, beta_h) -> c(x_h, beta_h)
    equivalent to tau_h -> tau_h/c leave (resp. change) the output in a way that fixes
    tau_h dtau_h exactly: sum W dW + sum beta dbeta + tau dtau = 0 and
    sum x dx + sum beta dbeta + tau dtau = 0, per head."""
    _, (x, fx, W, b, t, M, dO), fw, bw = _grads(16)
    for h in range(3):
        wb = (W[h] * bw["dW"][h]).sum() + (b[h] * bw["dbias"][h]).sum()
        xb = (x[:, :, h, :] * bw["dx_mid"][:, :, h, :]).sum() + (b[h] * bw["dbias"][h]).sum()
        scale = abs(t[h] * bw["dtau"][h]) + abs(wb) + 1e-300
        assert abs(wb + t[h] * bw["dtau"][h]) / scale < 1e-12
        assert abs(xb + t[h] * bw["dtau"][h]) / scale < 1e-12


def test_shift_invariance():
    """beta_h + c and W_h[k, :] + c shift every logit of a point equally."""
    _, _, _, bw = _grads(17)
    np.testing.assert_allclose(bw["dbias"].sum(axis=1), 0.0, atol=1e-12 * np.abs(bw["dbias"]).max())
    np.testing.assert_allclose(bw["dW"].sum(axis=2), 0.0, atol=1e-12 * np.abs(bw["dW"]).max())


def test_unnormalised_partials_then_finalize():
    """finalize=False gives (U, S); normalising afterwards equals the finalized slice,
    and the exchanged partial has H*G*(d+1) floats: 33,792 B at the paper's
    H=8, G=32, D=32 (App. G.4 quotes about 33 KB; the token block alone is 32 KB)."""
    wl = make_case(B=1, N=100, H=8, d=32, G=32, seed=18, backward=False)
    a = orc.slice_fwd(wl.x_mid, wl.fx, wl.W_slice, wl.bias, wl.tau, eps=wl.eps, finalize=True)
    u = orc.slice_fwd(wl.x_mid, wl.fx, wl.W_slice, wl.bias, wl.tau, eps=wl.eps, finalize=False)
    np.testing.assert_allclose(orc.slice_finalize(u["tokens"], u["wsum"], wl.eps), a["tokens"], rtol=1e-13)
    assert a["tokens"][0].size * 4 == 32 * 1024
    assert (u["tokens"][0].size + u["wsum"][0].size) * 4 == 33792


def test_point_chunking_does_not_change_results(monkeypatch):
    wl = make_case(B=2, N=77, H=2, d=4, G=5, seed=19)
    x, fx, W, b, t, M, dO = _case_arrays(wl)
    ref_f = orc.forward(x, fx, W, b, t, M, eps=wl.eps)
    ref_b = orc.backward(x, fx, W, b, t, M, dO, eps=wl.eps)
    monkeypatch.setattr(orc, "_CHUNK", 10)
    f = orc.forward(x, fx, W, b, t, M, eps=wl.eps)
    g = orc.backward(x, fx, W, b, t, M, dO, eps=wl.eps)
    for k in ("tokens", "out", "lse"):
        np.testing.assert_allclose(f[k], ref_f[k], rtol=1e-12, atol=1e-14)
    for k in ("dx_mid", "dfx", "dW", "dbias", "dtau", "dM"):
        np.testing.assert_allclose(g[k], ref_b[k], rtol=1e-11, atol=1e-13)


def test_head_and_point_subsets_match_full():
    """Subset evaluation (used at full sizes) agrees with the full computation."""
    wl = make_case(B=2, N=60, H=3, d=4, G=5, seed=20)
    x, fx, W, b, t, M, dO = _case_arrays(wl)
    full = orc.forward(x, fx, W, b, t, M, eps=wl.eps)
    pts = np.array([0, 7, 59])
    sub = orc.forward(x, fx, W, b, t, M, eps=wl.eps, heads=[1], points=pts)
    np.testing.assert_allclose(sub["tokens"][:, 1], full["tokens"][:, 1], rtol=1e-13)
    np.testing.assert_allclose(sub["out"][:, pts, 1], full["out"][:, pts, 1], rtol=1e-13)
    assert np.isnan(sub["out"][:, 1, 1]).all() and np.isnan(sub["tokens"][:, 0]).all()
    fb = orc.backward(x, fx, W, b, t, M, dO, eps=wl.eps)
    sb = orc.backward(x, fx, W, b, t, M, dO, eps=wl.eps, heads=[2])
    for k in ("dW", "dbias", "dtau", "dM"):
        np.testing.assert_allclose(sb[k][2], fb[k][2], rtol=1e-12)
