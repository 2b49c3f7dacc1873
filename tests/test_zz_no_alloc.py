"""fs_slice_fwd_noalloc (the slice forward on the library's fixed device scratch,
no workspace argument) against fs_slice_fwd with a caller workspace, both
through the C ABI.  The file name sorts last, so in a full run it executes
after every other test in the same process; it passes alone as well.

Tolerance: the test's usual per-tensor bound (fp32: normwise max relative
error 1e-4; bf16: relative L2 1e-2).  Both entry points run the same
deterministic kernels, so in practice the results agree bit for bit.
"""
import types

import pytest
import torch

from paper_2609_32525_gb300.workloads import make_case

from _parity import error, host, tol, upload

# (B, N, H, d, G, dtype): the tensor-core path (bf16, d = 32, G a multiple of
# 128) and the SIMT fp32 path, both within the fixed scratch.
CASES = [(1, 3000, 4, 32, 256, "bf16"), (2, 700, 2, 16, 40, "f32")]


@pytest.mark.gpu
@pytest.mark.parametrize("case", CASES, ids=lambda c: "B{}N{}H{}d{}G{}-{}".format(*c))
def test_no_alloc_matches_workspace_entry_point(lib, case):
    B, N, H, d, G, dt = case
    wl = make_case(B, N, H, d, G, dtype=dt, seed=500 + N, backward=False)
    dev = upload(wl)
    s = lib.shape_of(dev["x_mid"], G, wl.eps)
    assert 0 < lib.workspace_bytes(s, lib.FS_OP_SLICE_FWD) <= lib.FS_NOALLOC_SCRATCH_BYTES
    f32 = dict(dtype=torch.float32, device="cuda")

    ref = (torch.empty(B, H, G, d, **f32), torch.empty(B, H, G, **f32), torch.empty(B, H, N, **f32))
    ws = lib.workspace(s, lib.FS_OP_SLICE_FWD)
    lib.fs_slice_fwd(s, dev["x_mid"], dev["fx"], dev["W_slice"], dev["bias"], dev["tau"], *ref, True, ws)
    torch.cuda.synchronize()
    assert lib.fs_device_status(ws) == lib.FS_OK

    for _ in range(2):  # two calls in a row on the same scratch
        got = (torch.full((B, H, G, d), float("nan"), **f32), torch.full((B, H, G), float("nan"), **f32),
               torch.full((B, H, N), float("nan"), **f32))
        addr = lib.fs_slice_fwd_noalloc(s, dev["x_mid"], dev["fx"], dev["W_slice"], dev["bias"], dev["tau"], *got,
                                        True)
        torch.cuda.synchronize()
        assert addr != 0
        assert lib.device_status_at(addr) == lib.FS_OK
        for name, g, r in zip(("tokens", "wsum", "lse"), got, ref):
            e = error(host(g), host(r), dt)
            assert e <= tol(dt), f"{name}: error {e:.3e} against fs_slice_fwd"


def test_no_alloc_rejects_a_shape_beyond_its_scratch():
    """Host-side rejection, before any device call (runs without a GPU)."""
    from paper_2609_32525_gb300 import build

    build.build()
    from paper_2609_32525_gb300 import flashslice as lib

    null_stream = types.SimpleNamespace(cuda_stream=0)  # no torch CUDA stream without a GPU
    s = lib.make_shape(1, 1 << 20, 8, 32, 1024, lib.FS_BF16)
    assert lib.workspace_bytes(s, lib.FS_OP_SLICE_FWD) > lib.FS_NOALLOC_SCRATCH_BYTES
    with pytest.raises(lib.FlashSliceError) as err:
        lib.fs_slice_fwd_noalloc(s, None, None, None, None, None, None, None, None, True, null_stream)
    assert err.value.status == lib.FS_ERR_SCRATCH_TOO_SMALL
    assert "fixed scratch" in lib.status_string(lib.FS_ERR_SCRATCH_TOO_SMALL)
    with pytest.raises(lib.FlashSliceError) as err:
        lib.fs_slice_fwd_noalloc(lib.make_shape(0, 10, 1, 32, 8), None, None, None, None, None, None, None, None, True,
                                 null_stream)
    assert err.value.status == lib.FS_ERR_INVALID
