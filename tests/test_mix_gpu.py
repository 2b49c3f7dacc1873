"""GPU parity of the token mix alone (Eq. (1) with a constant core) and of its
backward, through fs_mix and fs_mix_bwd, against the oracle's mix and mix_bwd
on the same seeded fp32 inputs.  Slot counts cover one and several 64-slot
chunks with ragged tails, G % 4 != 0 (the 4-byte staging path) and G up to 1500;
every supported channel count d, B > 1 (dM sums over the batch)."""
import numpy as np
import pytest
import torch

from oracle import flashslice_oracle as orc

from _parity import host, max_rel, tol

pytestmark = pytest.mark.gpu

SHAPES = [  # (B, H, d, G)
    (1, 1, 16, 1),
    (2, 2, 32, 3),
    (1, 3, 64, 48),
    (2, 2, 32, 100),
    (3, 1, 16, 130),
    (1, 2, 32, 257),
    (1, 8, 32, 1024),
    (2, 2, 64, 1500),
]


@pytest.mark.parametrize("shp", SHAPES, ids=lambda s: "B{}H{}d{}G{}".format(*s))
def test_mix_and_its_backward(lib, shp):
    B, H, d, G = shp
    rng = np.random.default_rng(1000 + G)
    M = (np.eye(G)[None] + 0.1 * rng.standard_normal((H, G, G))).astype(np.float32)
    z = rng.standard_normal((B, H, G, d)).astype(np.float32)
    dzp = rng.standard_normal((B, H, G, d)).astype(np.float32)
    dev = {k: torch.from_numpy(v).cuda() for k, v in (("M", M), ("z", z), ("dzp", dzp))}
    s = lib.make_shape(B, 1, H, d, G, dtype=lib.FS_F32)
    zp, dz, dM = torch.empty_like(dev["z"]), torch.empty_like(dev["z"]), torch.empty_like(dev["M"])
    lib.fs_mix(s, dev["M"], dev["z"], zp)
    lib.fs_mix_bwd(s, dev["M"], dev["z"], dev["dzp"], dz, dM)
    torch.cuda.synchronize()
    ref = orc.mix(M, z)
    rb = orc.mix_bwd(M, z, dzp)
    for name, got, want in (("tokens_mixed", zp, ref), ("d_tokens", dz, rb["d_tokens"]), ("dM", dM, rb["dM"])):
        e = max_rel(host(got), want)
        print(f"PARITY mix B{B}H{H}d{d}G{G} {name} {e:.3e} tol {tol('f32'):.0e}")
        assert e <= tol("f32"), f"{name}: {e:.3e}"
