"""Pins of the oracle's NoTokenAttn core, the per-token channel map
z'[b,h,g,:] = Wc[h] z[b,h,g,:] (Sec. 2 after Eq. (1); Sec. 3 variants table), on CPU:

* the scalar-loop restatement (oracle/bruteforce.py) to 1e-12, forward and backward;
* central finite differences of both gradients;
* the identity map and the zero map;
* the exact identities <z', dz'> = <Wc, dWc> = <z, dz> (z' is linear in Wc and in z);
* it commutes with the slot mix (they act on different indices), and a NoTokenAttn
  layer (slice -> channel map -> deslice) with Wc = I equals the coupling with M = I.
"""
import numpy as np

from oracle import bruteforce
from oracle import flashslice_oracle as orc
from paper_2609_32525_gb300.workloads import make_case


def _draw(seed, B=2, H=3, G=5, d=4):
    rng = np.random.default_rng(seed)
    return rng.standard_normal((H, d, d)), rng.standard_normal((B, H, G, d)), rng.standard_normal((B, H, G, d))


def test_channel_map_matches_scalar_loops():
    Wc, z, dzp = _draw(1)
    B, H, G, d = z.shape
    np.testing.assert_allclose(orc.mix_channels(Wc, z), np.array(bruteforce.mix_channels(Wc, z, B, H, G, d)),
                               rtol=1e-12, atol=1e-12)
    bw = orc.mix_channels_bwd(Wc, z, dzp)
    dz, dWc = bruteforce.mix_channels_bwd(Wc, z, dzp, B, H, G, d)
    np.testing.assert_allclose(bw["d_tokens"], np.array(dz), rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(bw["dWc"], np.array(dWc), rtol=1e-12, atol=1e-12)


def test_channel_map_finite_differences():
    Wc, z, dzp = _draw(2)
    bw = orc.mix_channels_bwd(Wc, z, dzp)
    loss = lambda W_, z_: float((orc.mix_channels(W_, z_) * dzp).sum())
    h = 1e-6
    for name, p, g in (("dWc", Wc, bw["dWc"]), ("d_tokens", z, bw["d_tokens"])):
        fd = np.zeros_like(p)
        for i in np.ndindex(p.shape):
            old = p[i]
            p[i] = old + h
            lp = loss(Wc, z)
            p[i] = old - h
            lm = loss(Wc, z)
            p[i] = old
            fd[i] = (lp - lm) / (2 * h)
        assert np.linalg.norm(fd - g) / np.linalg.norm(g) < 1e-8, name


def test_identity_and_zero_maps():
    _, z, _ = _draw(3)
    H, d = z.shape[1], z.shape[3]
    eye = np.broadcast_to(np.eye(d), (H, d, d))
    np.testing.assert_array_equal(orc.mix_channels(eye, z), z)
    np.testing.assert_array_equal(orc.mix_channels(np.zeros((H, d, d)), z), np.zeros_like(z))


def test_linearity_identities():
    Wc, z, dzp = _draw(4)
    zp = orc.mix_channels(Wc, z)
    bw = orc.mix_channels_bwd(Wc, z, dzp)
    L = (zp * dzp).sum()
    np.testing.assert_allclose((Wc * bw["dWc"]).sum(), L, rtol=1e-12)
    np.testing.assert_allclose((z * bw["d_tokens"]).sum(), L, rtol=1e-12)


def test_commutes_with_the_slot_mix_and_reduces_to_the_identity_core():
    Wc, z, _ = _draw(5)
    B, H, G, d = z.shape
    M = np.random.default_rng(6).standard_normal((H, G, G))
    np.testing.assert_allclose(orc.mix(M, orc.mix_channels(Wc, z)), orc.mix_channels(Wc, orc.mix(M, z)),
                               rtol=1e-12, atol=1e-12)
    wl = make_case(B=1, N=50, H=2, d=4, G=6, seed=7, backward=False)
    eye_c = np.broadcast_to(np.eye(4), (2, 4, 4))
    eye_g = np.broadcast_to(np.eye(6), (2, 6, 6))
    s = orc.slice_fwd(wl.x_mid, wl.fx, wl.W_slice, wl.bias, wl.tau, eps=wl.eps)
    out_nt = orc.deslice_fwd(wl.x_mid, wl.W_slice, wl.bias, wl.tau, orc.mix_channels(eye_c, s["tokens"]))
    out_id = orc.forward(wl.x_mid, wl.fx, wl.W_slice, wl.bias, wl.tau, eye_g, eps=wl.eps)["out"]
    np.testing.assert_allclose(out_nt, out_id, rtol=1e-12, atol=1e-12)
