"""Host-side checks of the C-ABI library: it loads, exports every entry point the
header declares, and validates arguments before launching anything.  No GPU:
every call here fails validation (or only queries sizes) before any launch."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "flashslice.h")
LIB = os.path.join(ROOT, "paper_2609_32525_gb300", "libflashslice.so")


@pytest.fixture(scope="module")
def fs():
    if not os.path.exists(LIB):
        from paper_2609_32525_gb300 import build

        build.build()
    from paper_2609_32525_gb300 import flashslice

    return flashslice


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(fs_[a-z_]+)\s*\(", text)))


def test_header_declares_the_documented_entry_points():
    names = declared_functions()
    for n in ("fs_slice_fwd", "fs_mix", "fs_deslice_fwd", "fs_slice_bwd", "fs_deslice_bwd", "fs_mix_bwd",
              "fs_slice_finalize", "fs_workspace_bytes", "fs_device_status", "fs_status_string"):
        assert n in names


def test_library_exports_every_declared_symbol(fs):
    lib = ctypes.CDLL(LIB)
    for name in declared_functions():
        assert hasattr(lib, name), name
    assert set(fs.EXPORTED) <= set(declared_functions())


def test_status_strings(fs):
    for st in range(6):
        assert fs.status_string(st).startswith("FS_")
    assert "unknown" in fs.status_string(99)


def test_workspace_sizes(fs):
    s = fs.make_shape(1, 4096, 8, 32, 32)
    for op in (fs.FS_OP_SLICE_FWD, fs.FS_OP_DESLICE_FWD, fs.FS_OP_DESLICE_BWD, fs.FS_OP_SLICE_BWD, fs.FS_OP_STATS):
        assert fs.workspace_bytes(s, op) >= 256
    assert fs.workspace_bytes(fs.make_shape(1, 4096, 8, 32, 32), 99) == 0
    assert fs.workspace_bytes(fs.make_shape(0, 4096, 8, 32, 32), 0) == 0       # invalid
    assert fs.workspace_bytes(fs.make_shape(1, 4096, 8, 48, 32), 0) == 0       # unsupported d
    big = fs.workspace_bytes(fs.make_shape(1, 1 << 20, 8, 32, 1024), fs.FS_OP_SLICE_FWD)
    assert big >= (1 << 20) * 8 * 4  # at least the lse scratch


def _call_slice(fs, shape, ptrs, ws_ptr=16, ws_bytes=1 << 30):
    lib = fs._lib
    P = ctypes.c_void_p
    return lib.fs_slice_fwd(ctypes.byref(shape), *[P(p) if p else None for p in ptrs], None, 1, P(ws_ptr) if ws_ptr else None,
                            ws_bytes, None)


def test_validation_rejects_bad_arguments_without_launching(fs):
    good = [16 * (i + 1) for i in range(7)]  # fake aligned addresses, never dereferenced
    s = fs.make_shape(1, 100, 2, 32, 8)
    # null pointer
    assert _call_slice(fs, s, [0] + good[1:]) == fs.FS_ERR_INVALID
    # misaligned pointer
    assert _call_slice(fs, s, [good[0] + 4] + good[1:]) == fs.FS_ERR_INVALID
    # bad sizes
    for bad in (fs.make_shape(0, 100, 2, 32, 8), fs.make_shape(1, 0, 2, 32, 8), fs.make_shape(1, 100, 0, 32, 8),
                fs.make_shape(1, 100, 2, 32, 0), fs.make_shape(1, 100, 2, 32, 8, dtype=7),
                fs.make_shape(1, 100, 2, 32, 8, eps=-1.0), fs.make_shape(1, 100, 2, 32, 8, eps=float("nan"))):
        assert _call_slice(fs, bad, good) == fs.FS_ERR_INVALID
    # unsupported head width / slice count
    assert _call_slice(fs, fs.make_shape(1, 100, 2, 48, 8), good) == fs.FS_ERR_UNSUPPORTED
    assert _call_slice(fs, fs.make_shape(1, 100, 2, 32, 5000), good) == fs.FS_ERR_UNSUPPORTED
    # workspace missing or too small
    assert _call_slice(fs, s, good, ws_ptr=0) == fs.FS_ERR_INVALID
    assert _call_slice(fs, s, good, ws_bytes=8) == fs.FS_ERR_INVALID


def test_stats_validation(fs):
    """fs_stats checks its pointers, shape and workspace before any launch."""
    lib, P = fs._lib, ctypes.c_void_p
    s = fs.make_shape(1, 100, 2, 32, 8)
    ptrs = [P(16 * (i + 1)) for i in range(5)]  # fake aligned addresses, never dereferenced

    def call(shape, args, ws=P(16), ws_bytes=1 << 30):
        return lib.fs_stats(ctypes.byref(shape), *args, ws, ws_bytes, None)

    for i in range(5):
        assert call(s, ptrs[:i] + [None] + ptrs[i + 1:]) == fs.FS_ERR_INVALID
    assert call(fs.make_shape(1, 0, 2, 32, 8), ptrs) == fs.FS_ERR_INVALID
    assert call(fs.make_shape(1, 100, 2, 48, 8), ptrs) == fs.FS_ERR_UNSUPPORTED
    assert call(s, ptrs, ws=None) == fs.FS_ERR_INVALID
    assert call(s, ptrs, ws_bytes=fs.workspace_bytes(s, fs.FS_OP_STATS) - 1) == fs.FS_ERR_INVALID


def test_mix_rejects_in_place(fs):
    s = fs.make_shape(1, 100, 2, 32, 8)
    P = ctypes.c_void_p
    assert fs._lib.fs_mix(ctypes.byref(s), P(16), P(32), P(32), None) == fs.FS_ERR_INVALID
    assert fs._lib.fs_device_status(None, None) == fs.FS_ERR_INVALID


def test_mix_calls_reject_partly_overlapping_buffers(fs):
    """The mixes and their backward read every input while writing: an output that
    shares any byte with an input (or another output) is rejected before any
    launch.  Fake 16-byte-aligned addresses, never dereferenced: every call below
    fails validation."""
    lib, P = fs._lib, ctypes.c_void_p
    B, H, d, G = 1, 2, 32, 8
    s = fs.make_shape(B, 100, H, d, G)
    tb = B * H * G * d * 4        # tokens [B,H,G,d] fp32
    mb = H * G * G * 4            # M [H,G,G]
    wb = H * d * d * 4            # Wc [H,d,d]
    base = 1 << 20
    M, tok = base, base + 4 * tb
    # the output starts inside tokens (tail overlap) or ends inside it (head overlap)
    for out in (tok + 16, tok - tb + 16):
        assert lib.fs_mix(ctypes.byref(s), P(M), P(tok), P(out), None) == fs.FS_ERR_INVALID
        assert lib.fs_mix_channels(ctypes.byref(s), P(M), P(tok), P(out), None) == fs.FS_ERR_INVALID
    # the output overlaps M / Wc
    assert lib.fs_mix(ctypes.byref(s), P(M), P(tok), P(M + mb - 16), None) == fs.FS_ERR_INVALID
    assert lib.fs_mix_channels(ctypes.byref(s), P(M), P(tok), P(M + wb - 16), None) == fs.FS_ERR_INVALID
    # backward: d_tokens over d_tokens_mixed, dM over tokens, the two outputs over each other
    dzp, dz, dM = base + 8 * tb, base + 12 * tb, base + 16 * tb
    for args in ((M, tok, dzp, dzp + 16, dM), (M, tok, dzp, dz, tok + 16), (M, tok, dzp, dz, dz + 16)):
        assert lib.fs_mix_bwd(ctypes.byref(s), *[P(a) for a in args], None) == fs.FS_ERR_INVALID
        assert lib.fs_mix_channels_bwd(ctypes.byref(s), *[P(a) for a in args], None) == fs.FS_ERR_INVALID


def test_path_query(fs):
    assert fs.path_for_shape(fs.make_shape(1, 100, 2, 48, 8)) == -1
    assert fs.path_for_shape(fs.make_shape(1, 100, 2, 32, 8, dtype=fs.FS_F32)) == 0
    assert fs.forward_launch_count(fs.make_shape(1, 100, 2, 32, 8)) >= 3


def test_backward_launch_count(fs):
    assert fs.backward_launch_count(fs.make_shape(1, 100, 2, 48, 8)) == -1
    # the fp32 SIMT backward: 5 + 2 + 5 kernels, and the statistics pass once per
    # backward call when no lse is given
    s = fs.make_shape(1, 100, 2, 32, 8, dtype=fs.FS_F32)
    assert fs.backward_launch_count(s, True) == 12
    assert fs.backward_launch_count(s, False) == 14


def test_coupling_bwd_launch_count_and_overlap_checks(fs):
    """fs_coupling_bwd: on the SIMT backward it makes one fused pass pair (d z' partials
    and their reduction, the mix backward's two kernels, the dU, dS prologue, the point
    and slot passes, two reductions: 9 kernels, plus the statistics once when no lse
    is given) where the three calls make 12; outputs overlapping M, tokens,
    tokens_mixed or each other are rejected before any launch (fake aligned addresses,
    never read)."""
    s = fs.make_shape(1, 100, 2, 32, 8, dtype=fs.FS_F32)
    assert fs.coupling_bwd_launch_count(s, True) == 9
    assert fs.coupling_bwd_launch_count(s, False) == 10
    assert fs.backward_launch_count(s, True) == 12
    assert fs.coupling_bwd_launch_count(fs.make_shape(1, 100, 2, 48, 8)) == -1
    lib, P = fs._lib, ctypes.c_void_p
    B, N, H, d, G = 1, 100, 2, 32, 8
    tb, mb, pb = B * H * G * d * 4, H * G * G * 4, B * N * H * d * 4
    base = 1 << 24
    addr = [base + i * (1 << 20) for i in range(20)]
    ws = 1 << 30
    nbytes = fs.workspace_bytes(s, fs.FS_OP_COUPLING_BWD)
    assert nbytes > 0
    # x, fx, W, bias, tau, M, tokens, wsum, tokens_mixed, lse, dout | dzm, dz, dx, dfx, dW, db, dt, dM
    ins, outs = addr[:11], addr[11:19]
    M, tokens, tokens_mixed = ins[5], ins[6], ins[8]

    def call(o):
        return lib.fs_coupling_bwd(ctypes.byref(s), *[P(a) for a in ins], *[P(a) for a in o], 0, P(ws), nbytes, None)

    for k, target in ((0, tokens), (1, tokens_mixed), (7, M)):  # d_tokens_mixed, d_tokens, dM over an input
        o = list(outs)
        o[k] = target + 16
        assert call(o) == fs.FS_ERR_INVALID
    o = list(outs)
    o[1] = o[0] + 16  # d_tokens over d_tokens_mixed
    assert call(o) == fs.FS_ERR_INVALID
    assert lib.fs_coupling_bwd(ctypes.byref(s), *[P(a) for a in ins], *[P(a) for a in outs], 0, P(ws), nbytes - 1,
                               None) == fs.FS_ERR_INVALID
