"""Python binding of libflashslice.so (include/flashslice.h): argument marshalling only.

Every function named fs_* here calls the C entry point of the same name with
the device pointers of torch tensors and the current CUDA stream, and raises
FlashSliceError on a non-FS_OK status.  All compute happens in the library's
CUDA kernels; there is no fallback of any kind.  Importing this module loads
the library and fails loudly if it has not been built
(`python -m paper_2609_32525_gb300.build`).

Tensor conventions (see the header for the full contract):
  x_mid, fx, out, dout, dx_mid, dfx : [B,N,H,d] float32 or bfloat16, contiguous
  W_slice [H,d,G], bias [H,G], tau [H], M [H,G,G]            float32
  tokens, tokens_mixed, d_tokens*  [B,H,G,d], wsum [B,H,G], lse [B,H,N]  float32
"""
from __future__ import annotations

import ctypes
import os

import torch

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libflashslice.so")
if not os.path.exists(_LIB_PATH):
    raise ImportError(f"{_LIB_PATH} is missing: build it with `python -m paper_2609_32525_gb300.build` "
                      "(the library has no CPU fallback)")
_lib = ctypes.CDLL(_LIB_PATH)

FS_OK, FS_ERR_INVALID, FS_ERR_UNSUPPORTED, FS_ERR_CUDA, FS_ERR_TIMEOUT, FS_ERR_BAD_TAU, FS_ERR_SCRATCH_TOO_SMALL = range(7)
FS_NOALLOC_SCRATCH_BYTES = 16 << 20
FS_F32, FS_BF16 = 0, 1
FS_DOT_BF16, FS_DOT_BF16X2 = 0, 1
FS_OP_SLICE_FWD, FS_OP_DESLICE_FWD, FS_OP_DESLICE_BWD, FS_OP_SLICE_BWD, FS_OP_STATS, FS_OP_COUPLING_BWD = range(6)

EXPORTED = ("fs_workspace_bytes", "fs_slice_fwd", "fs_slice_finalize", "fs_mix", "fs_deslice_fwd",
            "fs_deslice_bwd", "fs_mix_bwd", "fs_slice_bwd", "fs_device_status", "fs_status_string",
            "fs_path_for_shape", "fs_backward_path_for_shape", "fs_forward_launch_count", "fs_backward_launch_count",
            "fs_slice_fwd_noalloc", "fs_slice_fwd_lse", "fs_mix_channels", "fs_mix_channels_bwd", "fs_stats",
            "fs_coupling_bwd", "fs_coupling_bwd_launch_count")


class fs_shape(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int64), ("N", ctypes.c_int64), ("H", ctypes.c_int32), ("d", ctypes.c_int32),
                ("G", ctypes.c_int32), ("dtype", ctypes.c_int32), ("eps", ctypes.c_float), ("dot", ctypes.c_int32)]


class FlashSliceError(RuntimeError):
    def __init__(self, fn, status):
        self.status = status
        super().__init__(f"{fn}: {_lib.fs_status_string(status).decode()}")


_P = ctypes.c_void_p
_S = ctypes.POINTER(fs_shape)
_I = ctypes.c_int
_Z = ctypes.c_size_t
_sig = {
    "fs_workspace_bytes": (_Z, [_S, _I]),
    "fs_slice_fwd": (_I, [_S, _P, _P, _P, _P, _P, _P, _P, _P, _I, _P, _Z, _P]),
    "fs_slice_fwd_lse": (_I, [_S, _P, _P, _P, _P, _P, _P, _P, _P, _I, _P, _Z, _P]),
    "fs_slice_finalize": (_I, [_S, _P, _P, _P]),
    "fs_stats": (_I, [_S, _P, _P, _P, _P, _P, _P, _Z, _P]),
    "fs_mix_channels": (_I, [_S, _P, _P, _P, _P]),
    "fs_mix_channels_bwd": (_I, [_S, _P, _P, _P, _P, _P, _P]),
    "fs_mix": (_I, [_S, _P, _P, _P, _P]),
    "fs_deslice_fwd": (_I, [_S, _P, _P, _P, _P, _P, _P, _P, _P, _Z, _P]),
    "fs_deslice_bwd": (_I, [_S, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _I, _P, _Z, _P]),
    "fs_mix_bwd": (_I, [_S, _P, _P, _P, _P, _P, _P]),
    "fs_slice_bwd": (_I, [_S, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _I, _P, _Z, _P]),
    "fs_device_status": (_I, [_P, _P]),
    "fs_status_string": (ctypes.c_char_p, [_I]),
    "fs_path_for_shape": (_I, [_S]),
    "fs_backward_path_for_shape": (_I, [_S]),
    "fs_forward_launch_count": (_I, [_S]),
    "fs_backward_launch_count": (_I, [_S, _I]),
    "fs_coupling_bwd_launch_count": (_I, [_S, _I]),
    "fs_coupling_bwd": (_I, [_S] + [_P] * 11 + [_P] * 8 + [_I, _P, _Z, _P]),
    "fs_slice_fwd_noalloc": (_I, [_S, _P, _P, _P, _P, _P, _P, _P, _P, _I, ctypes.POINTER(_P), _P]),
}
for _name, (_res, _args) in _sig.items():
    _f = getattr(_lib, _name)
    _f.restype = _res
    _f.argtypes = _args


def make_shape(B, N, H, d, G, dtype=FS_F32, eps=1e-5, dot=None) -> fs_shape:
    """dot: FS_DOT_BF16 (default) or FS_DOT_BF16X2 (see the header)."""
    if isinstance(dtype, torch.dtype):
        dtype = FS_BF16 if dtype == torch.bfloat16 else FS_F32
    return fs_shape(int(B), int(N), int(H), int(d), int(G), int(dtype), float(eps),
                    int(FS_DOT_BF16 if dot is None else dot))


def shape_of(x_mid: torch.Tensor, G: int, eps: float = 1e-5, dot=None) -> fs_shape:
    B, N, H, d = x_mid.shape
    return make_shape(B, N, H, d, G, x_mid.dtype, eps, dot)


def _ptr(t):
    if t is None:
        return None
    if not t.is_contiguous():
        raise ValueError("flashslice tensors must be contiguous")
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream=None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _check(fn, st):
    if st != FS_OK:
        raise FlashSliceError(fn, st)


def workspace_bytes(shape: fs_shape, op: int) -> int:
    return int(_lib.fs_workspace_bytes(ctypes.byref(shape), op))


def workspace(shape: fs_shape, op: int, device="cuda") -> torch.Tensor:
    """Scratch for one op, allocated through torch (the library never allocates).
    Its status word starts at FS_OK, so a scratch no call has used yet reads clean."""
    n = max(16, workspace_bytes(shape, op))
    ws = torch.empty(n, dtype=torch.uint8, device=device)
    ws[:16].zero_()
    return ws


def path_for_shape(shape: fs_shape) -> int:
    return int(_lib.fs_path_for_shape(ctypes.byref(shape)))


def backward_path_for_shape(shape: fs_shape) -> int:
    return int(_lib.fs_backward_path_for_shape(ctypes.byref(shape)))


def forward_launch_count(shape: fs_shape) -> int:
    return int(_lib.fs_forward_launch_count(ctypes.byref(shape)))


def backward_launch_count(shape: fs_shape, lse_given: bool = True) -> int:
    return int(_lib.fs_backward_launch_count(ctypes.byref(shape), int(bool(lse_given))))


def coupling_bwd_launch_count(shape: fs_shape, lse_given: bool = True) -> int:
    return int(_lib.fs_coupling_bwd_launch_count(ctypes.byref(shape), int(bool(lse_given))))


def status_string(st: int) -> str:
    return _lib.fs_status_string(st).decode()


def fs_slice_fwd(shape, x_mid, fx, W_slice, bias, tau, tokens, wsum, lse, finalize, ws, stream=None):
    st = _lib.fs_slice_fwd(ctypes.byref(shape), _ptr(x_mid), _ptr(fx), _ptr(W_slice), _ptr(bias), _ptr(tau),
                           _ptr(tokens), _ptr(wsum), _ptr(lse), int(bool(finalize)), _ptr(ws), ws.numel(),
                           _stream(stream))
    _check("fs_slice_fwd", st)


def fs_stats(shape, x_mid, W_slice, bias, tau, lse, ws, stream=None):
    st = _lib.fs_stats(ctypes.byref(shape), _ptr(x_mid), _ptr(W_slice), _ptr(bias), _ptr(tau), _ptr(lse), _ptr(ws),
                       ws.numel(), _stream(stream))
    _check("fs_stats", st)


def fs_slice_fwd_lse(shape, x_mid, fx, W_slice, bias, tau, lse, tokens, wsum, finalize, ws, stream=None):
    st = _lib.fs_slice_fwd_lse(ctypes.byref(shape), _ptr(x_mid), _ptr(fx), _ptr(W_slice), _ptr(bias), _ptr(tau),
                               _ptr(lse), _ptr(tokens), _ptr(wsum), int(bool(finalize)), _ptr(ws), ws.numel(),
                               _stream(stream))
    _check("fs_slice_fwd_lse", st)


def fs_mix_channels(shape, Wc, tokens, tokens_mixed, stream=None):
    _check("fs_mix_channels", _lib.fs_mix_channels(ctypes.byref(shape), _ptr(Wc), _ptr(tokens), _ptr(tokens_mixed),
                                                   _stream(stream)))


def fs_mix_channels_bwd(shape, Wc, tokens, d_tokens_mixed, d_tokens, dWc, stream=None):
    _check("fs_mix_channels_bwd", _lib.fs_mix_channels_bwd(ctypes.byref(shape), _ptr(Wc), _ptr(tokens),
                                                           _ptr(d_tokens_mixed), _ptr(d_tokens), _ptr(dWc),
                                                           _stream(stream)))


def fs_slice_finalize(shape, tokens, wsum, stream=None):
    _check("fs_slice_finalize", _lib.fs_slice_finalize(ctypes.byref(shape), _ptr(tokens), _ptr(wsum),
                                                       _stream(stream)))


def fs_mix(shape, M, tokens, tokens_mixed, stream=None):
    _check("fs_mix", _lib.fs_mix(ctypes.byref(shape), _ptr(M), _ptr(tokens), _ptr(tokens_mixed), _stream(stream)))


def fs_deslice_fwd(shape, x_mid, W_slice, bias, tau, tokens_mixed, lse, out, ws, stream=None):
    st = _lib.fs_deslice_fwd(ctypes.byref(shape), _ptr(x_mid), _ptr(W_slice), _ptr(bias), _ptr(tau),
                             _ptr(tokens_mixed), _ptr(lse), _ptr(out), _ptr(ws), ws.numel(), _stream(stream))
    _check("fs_deslice_fwd", st)


def fs_deslice_bwd(shape, x_mid, W_slice, bias, tau, tokens_mixed, lse, dout, d_tokens_mixed, dx_mid, dW, dbias,
                   dtau, accumulate, ws, stream=None):
    st = _lib.fs_deslice_bwd(ctypes.byref(shape), _ptr(x_mid), _ptr(W_slice), _ptr(bias), _ptr(tau),
                             _ptr(tokens_mixed), _ptr(lse), _ptr(dout), _ptr(d_tokens_mixed), _ptr(dx_mid),
                             _ptr(dW), _ptr(dbias), _ptr(dtau), int(bool(accumulate)), _ptr(ws), ws.numel(),
                             _stream(stream))
    _check("fs_deslice_bwd", st)


def fs_mix_bwd(shape, M, tokens, d_tokens_mixed, d_tokens, dM, stream=None):
    st = _lib.fs_mix_bwd(ctypes.byref(shape), _ptr(M), _ptr(tokens), _ptr(d_tokens_mixed), _ptr(d_tokens),
                         _ptr(dM), _stream(stream))
    _check("fs_mix_bwd", st)


def fs_slice_bwd(shape, x_mid, fx, W_slice, bias, tau, tokens, wsum, lse, d_tokens, dx_mid, dfx, dW, dbias, dtau,
                 accumulate, ws, stream=None):
    st = _lib.fs_slice_bwd(ctypes.byref(shape), _ptr(x_mid), _ptr(fx), _ptr(W_slice), _ptr(bias), _ptr(tau),
                           _ptr(tokens), _ptr(wsum), _ptr(lse), _ptr(d_tokens), _ptr(dx_mid), _ptr(dfx), _ptr(dW),
                           _ptr(dbias), _ptr(dtau), int(bool(accumulate)), _ptr(ws), ws.numel(), _stream(stream))
    _check("fs_slice_bwd", st)


def fs_coupling_bwd(shape, x_mid, fx, W_slice, bias, tau, M, tokens, wsum, tokens_mixed, lse, dout, d_tokens_mixed,
                    d_tokens, dx_mid, dfx, dW, dbias, dtau, dM, accumulate, ws, stream=None):
    st = _lib.fs_coupling_bwd(ctypes.byref(shape), _ptr(x_mid), _ptr(fx), _ptr(W_slice), _ptr(bias), _ptr(tau),
                              _ptr(M), _ptr(tokens), _ptr(wsum), _ptr(tokens_mixed), _ptr(lse), _ptr(dout),
                              _ptr(d_tokens_mixed), _ptr(d_tokens), _ptr(dx_mid), _ptr(dfx), _ptr(dW), _ptr(dbias),
                              _ptr(dtau), _ptr(dM), int(bool(accumulate)), _ptr(ws), ws.numel(), _stream(stream))
    _check("fs_coupling_bwd", st)


def fs_device_status(ws, stream=None) -> int:
    return int(_lib.fs_device_status(_ptr(ws), _stream(stream)))


def fs_slice_fwd_noalloc(shape, x_mid, fx, W_slice, bias, tau, tokens, wsum, lse, finalize, stream=None) -> int:
    """fs_slice_fwd on the library's fixed device scratch (no workspace argument, nothing
    allocated).  Returns the scratch's device address, for device_status_at."""
    addr = _P()
    st = _lib.fs_slice_fwd_noalloc(ctypes.byref(shape), _ptr(x_mid), _ptr(fx), _ptr(W_slice), _ptr(bias),
                                   _ptr(tau), _ptr(tokens), _ptr(wsum), _ptr(lse), int(bool(finalize)),
                                   ctypes.byref(addr), _stream(stream))
    _check("fs_slice_fwd_noalloc", st)
    return int(addr.value)


def device_status_at(addr: int, stream=None) -> int:
    """fs_device_status of a scratch given by its device address."""
    return int(_lib.fs_device_status(_P(addr), _stream(stream)))


# ---- convenience: one coupling, buffers allocated through torch ----------------------------


class Coupling:
    """Allocates the outputs and scratch of one slice -> mix -> deslice coupling
    (forward, and backward when asked) once, then runs it through the C ABI."""

    def __init__(self, B, N, H, d, G, dtype=torch.bfloat16, eps=1e-5, backward=False, device="cuda", dot=None):
        # A coupling that will be differentiated defaults to the split products
        # (FS_DOT_BF16X2): the temperature gradient is a near-cancelling sum that
        # bf16 tokens cannot resolve.
        if dot is None:
            dot = FS_DOT_BF16X2 if backward else FS_DOT_BF16
        self.shape = make_shape(B, N, H, d, G, dtype, eps, dot)
        self.dtype = dtype
        f32 = dict(dtype=torch.float32, device=device)
        self.tokens = torch.empty(B, H, G, d, **f32)
        self.wsum = torch.empty(B, H, G, **f32)
        self.lse = torch.empty(B, H, N, **f32)
        self.tokens_mixed = torch.empty(B, H, G, d, **f32)
        self.out = torch.empty(B, N, H, d, dtype=dtype, device=device)
        self.ws_slice = workspace(self.shape, FS_OP_SLICE_FWD, device)
        self.ws_deslice = workspace(self.shape, FS_OP_DESLICE_FWD, device)
        if backward:
            self.d_tokens_mixed = torch.empty(B, H, G, d, **f32)
            self.d_tokens = torch.empty(B, H, G, d, **f32)
            self.dx_mid = torch.empty(B, N, H, d, dtype=dtype, device=device)
            self.dfx = torch.empty(B, N, H, d, dtype=dtype, device=device)
            self.dW = torch.empty(H, d, G, **f32)
            self.dbias = torch.empty(H, G, **f32)
            self.dtau = torch.empty(H, **f32)
            self.dM = torch.empty(H, G, G, **f32)
            self.ws_dbwd = workspace(self.shape, FS_OP_DESLICE_BWD, device)
            self.ws_sbwd = workspace(self.shape, FS_OP_SLICE_BWD, device)
            self.ws_cbwd = workspace(self.shape, FS_OP_COUPLING_BWD, device)

    def forward(self, x_mid, fx, W_slice, bias, tau, M, stream=None):
        s = self.shape
        fs_slice_fwd(s, x_mid, fx, W_slice, bias, tau, self.tokens, self.wsum, self.lse, True, self.ws_slice, stream)
        fs_mix(s, M, self.tokens, self.tokens_mixed, stream)
        fs_deslice_fwd(s, x_mid, W_slice, bias, tau, self.tokens_mixed, self.lse, self.out, self.ws_deslice, stream)
        return self.out

    def backward(self, x_mid, fx, W_slice, bias, tau, M, dout, stream=None, fused=True):
        """fused: one fs_coupling_bwd call; else fs_deslice_bwd, fs_mix_bwd, fs_slice_bwd."""
        s = self.shape
        if fused:
            fs_coupling_bwd(s, x_mid, fx, W_slice, bias, tau, M, self.tokens, self.wsum, self.tokens_mixed, self.lse,
                            dout, self.d_tokens_mixed, self.d_tokens, self.dx_mid, self.dfx, self.dW, self.dbias,
                            self.dtau, self.dM, False, self.ws_cbwd, stream)
        else:
            fs_deslice_bwd(s, x_mid, W_slice, bias, tau, self.tokens_mixed, self.lse, dout, self.d_tokens_mixed,
                           self.dx_mid, self.dW, self.dbias, self.dtau, False, self.ws_dbwd, stream)
            fs_mix_bwd(s, M, self.tokens, self.d_tokens_mixed, self.d_tokens, self.dM, stream)
            fs_slice_bwd(s, x_mid, fx, W_slice, bias, tau, self.tokens, self.wsum, self.lse, self.d_tokens,
                         self.dx_mid, self.dfx, self.dW, self.dbias, self.dtau, True, self.ws_sbwd, stream)
        return {"dx_mid": self.dx_mid, "dfx": self.dfx, "dW": self.dW, "dbias": self.dbias, "dtau": self.dtau,
                "dM": self.dM}

    def device_status(self, stream=None):
        worst = FS_OK
        for ws in (self.ws_slice, self.ws_deslice) + (
                (self.ws_dbwd, self.ws_sbwd, self.ws_cbwd) if hasattr(self, "ws_dbwd") else ()):
            st = fs_device_status(ws, stream)
            worst = worst or st
        return worst


class ShardedCoupling:
    """The local compute of a point-sharded coupling (App. G.4) for
    sharding.sharded_forward / sharding.sharded_backward: this rank's points of
    every batch, x_mid and fx [B, n_local, H, d], through the C ABI.  The slice
    keeps its numerators unnormalised (finalize = 0) until they are summed over
    ranks; the backward's two calls add into the same dx_mid, dW, dbias, dtau."""

    def __init__(self, B, n_local, H, d, G, x_mid, fx, W_slice, bias, tau, M, dtype=torch.bfloat16, eps=1e-5,
                 dout=None, device="cuda", dot=None):
        self.c = Coupling(B, n_local, H, d, G, dtype, eps, backward=dout is not None, device=device, dot=dot)
        self.x, self.fx, self.W, self.bias, self.tau, self.M, self.dout = x_mid, fx, W_slice, bias, tau, M, dout

    def slice_partials(self):
        c = self.c
        fs_slice_fwd(c.shape, self.x, self.fx, self.W, self.bias, self.tau, c.tokens, c.wsum, c.lse, False,
                     c.ws_slice)
        return c.tokens, c.wsum

    def finalize(self, U, S):
        fs_slice_finalize(self.c.shape, U, S)
        return U

    def mix(self, tokens):
        fs_mix(self.c.shape, self.M, tokens, self.c.tokens_mixed)
        return self.c.tokens_mixed

    def deslice(self, tokens_mixed):
        c = self.c
        fs_deslice_fwd(c.shape, self.x, self.W, self.bias, self.tau, tokens_mixed, c.lse, c.out, c.ws_deslice)
        return c.out

    def deslice_bwd(self):
        c = self.c
        fs_deslice_bwd(c.shape, self.x, self.W, self.bias, self.tau, c.tokens_mixed, c.lse, self.dout,
                       c.d_tokens_mixed, c.dx_mid, c.dW, c.dbias, c.dtau, False, c.ws_dbwd)
        return c.d_tokens_mixed

    def mix_bwd(self, d_tokens_mixed):
        c = self.c
        fs_mix_bwd(c.shape, self.M, c.tokens, d_tokens_mixed, c.d_tokens, c.dM)
        return c.d_tokens, c.dM

    def slice_bwd(self, d_tokens):
        c = self.c
        fs_slice_bwd(c.shape, self.x, self.fx, self.W, self.bias, self.tau, c.tokens, c.wsum, c.lse, d_tokens,
                     c.dx_mid, c.dfx, c.dW, c.dbias, c.dtau, True, c.ws_sbwd)
        return c.dW, c.dbias, c.dtau
