"""fp64 CPU oracle for Transolver's slice -> token mix -> deslice coupling.

TEST INFRASTRUCTURE ONLY.  This module is the independent reference that the
CUDA library is checked against.  Only the test-suite, the smoke check and the
CPU-baseline leg of the benchmark may import it; the library itself never does
and shares no code with it.

It is the *materialised* formulation written out plainly: for every (batch,
head) block the slice-weight matrix w (N x G) is formed explicitly, the slice
and deslice are matrix products with it, and the backward pass materialises
dw and da and applies the full softmax Jacobian-vector product.  numpy matmul
is the only library primitive used for the contractions; nothing is fused or
reordered beyond what the definitions below state.  Points may be processed in
chunks purely to bound memory (a sum over points split into partial sums);
that changes memory use, not the formula.

Notation (paper Sec. 2 "The Transolver layer" and Appendix G.1 "Single-tile
kernels"), per batch b and head h:
    x   = x_mid[b, :, h, :]             (N x d)   projection feeding the logits
    f   = fx[b, :, h, :]                (N x d)   projected values v_i / f_i
    W   = W_slice[h]                    (d x G)   slice projection
    beta= bias[h]                       (G)
    tau = tau[h]                                  learned temperature
    a   = (x W + beta) / tau            (N x G)   temperature-scaled logits
    w   = softmax over g of a           (N x G)   slice weights (partition of unity)
    S_g = sum_n w_ng                    (G)       weight sums  (s_g in App. G.1)
    U_g = sum_n w_ng f_n                (G x d)   token numerators (z^num)
    z_g = U_g / (S_g + eps)             (G x d)   tokens
    z'  = M z                           (G x d)   constant G x G token mix, the
                                                   core A of Eq. (1) acting on the
                                                   slot index: z'_g = sum_h A_gh z_h
    out_n = sum_g w_ng z'_g             (N x d)   deslice (tied weights)
Statistics: lse_n = log sum_g exp(a_ng) (natural log), so w = exp(a - lse).

Readings of the paper used here (all listed with their justification in the
design notes of the repository): eps is added to S (App. G.1 gives z^num/(s+eps)),
default 1e-5; W and the bias are per head; the mixer is per head and shared over
the batch, so dM sums over b; the temperature gradient follows App. G.2
("Temperature gradients"): dL/dtau = -sum_{n,g} dL/da_ng * a_ng / tau.
"""
from __future__ import annotations

import numpy as np

DEFAULT_EPS = 1e-5
# Points per chunk: bounds the materialised (chunk x G) fp64 matrices.
_CHUNK = 1 << 16


def _f64(a):
    return np.asarray(a, dtype=np.float64)


def logits(x, W, beta, tau):
    """Temperature-scaled slice logits a = (x W + beta) / tau (Sec. 2, App. G.1)."""
    return (_f64(x) @ _f64(W) + _f64(beta)[None, :]) / float(tau)


def softmax_rows(a):
    """Row softmax over the slot axis and its log-sum-exp.

    Returns (w, lse) with w_ng = exp(a_ng - lse_n).  The maximum is subtracted
    only for floating-point safety; it cancels mathematically.
    """
    m = a.max(axis=1, keepdims=True)
    e = np.exp(a - m)
    l = e.sum(axis=1, keepdims=True)
    return e / l, (m + np.log(l))[:, 0]


def _shape(x_mid, W_slice):
    B, N, H, d = x_mid.shape
    G = W_slice.shape[2]
    return B, N, H, d, G


def _heads(H, heads):
    return list(range(H)) if heads is None else list(heads)


def slice_fwd(x_mid, fx, W_slice, bias, tau, eps=DEFAULT_EPS, finalize=True, heads=None):
    """Slice operator (Sec. 2; App. G.1): tokens, weight sums and statistics.

    Returns dict with
      tokens [B,H,G,d]: z = U/(S+eps) if finalize else the numerators U
      wsum   [B,H,G]  : S
      lse    [B,N,H]  : log-sum-exp of the logits per point and head
    Heads not in `heads` are left as NaN (used to bound cost at large sizes).
    """
    B, N, H, d, G = _shape(x_mid, W_slice)
    tokens = np.full((B, H, G, d), np.nan)
    wsum = np.full((B, H, G), np.nan)
    lse = np.full((B, N, H), np.nan)
    for b in range(B):
        for h in _heads(H, heads):
            U = np.zeros((G, d))
            S = np.zeros(G)
            for n0 in range(0, N, _CHUNK):
                n1 = min(N, n0 + _CHUNK)
                a = logits(x_mid[b, n0:n1, h, :], W_slice[h], bias[h], tau[h])
                w, l = softmax_rows(a)
                U += w.T @ _f64(fx[b, n0:n1, h, :])
                S += w.sum(axis=0)
                lse[b, n0:n1, h] = l
            tokens[b, h] = U / (S + eps)[:, None] if finalize else U
            wsum[b, h] = S
    return {"tokens": tokens, "wsum": wsum, "lse": lse}


def slice_finalize(tokens_unnormalised, wsum, eps=DEFAULT_EPS):
    """Column normalisation applied after partial numerators are combined (App. G.1)."""
    return _f64(tokens_unnormalised) / (_f64(wsum) + eps)[..., None]


def mix(M, tokens):
    """Constant token mix z'_g = sum_h M_gh z_h per (b, head): the core of Eq. (1)."""
    M = _f64(M)
    tokens = _f64(tokens)
    return np.einsum("hgk,bhkc->bhgc", M, tokens)


def deslice_fwd(x_mid, W_slice, bias, tau, tokens_mixed, heads=None, points=None):
    """Deslice with tied weights: out_n = sum_g w_ng z'_g (Sec. 2; App. G.1).

    `points` optionally restricts the output to a sorted index array of points
    (other rows NaN) so that large workloads can be checked on a sample.
    """
    B, N, H, d, G = _shape(x_mid, W_slice)
    out = np.full((B, N, H, d), np.nan)
    idx = np.arange(N) if points is None else np.asarray(points)
    for b in range(B):
        for h in _heads(H, heads):
            for c0 in range(0, len(idx), _CHUNK):
                sel = idx[c0:c0 + _CHUNK]
                a = logits(x_mid[b, sel, h, :], W_slice[h], bias[h], tau[h])
                w, _ = softmax_rows(a)
                out[b, sel, h, :] = w @ _f64(tokens_mixed[b, h])
    return out


def forward(x_mid, fx, W_slice, bias, tau, M, eps=DEFAULT_EPS, heads=None, points=None):
    """Slice -> mix -> deslice for one physics-attention coupling."""
    s = slice_fwd(x_mid, fx, W_slice, bias, tau, eps, True, heads)
    tm = mix(M, s["tokens"])
    out = deslice_fwd(x_mid, W_slice, bias, tau, tm, heads, points)
    return {"tokens": s["tokens"], "wsum": s["wsum"], "lse": s["lse"],
            "tokens_mixed": tm, "out": out}


# --------------------------------------------------------------------------
# Backward.  Chain rule through the definitions above, per (b, h):
#   dz'_g  = sum_n w_ng dO_n                    (deslice, value path)
#   dw^D_ng = dO_n . z'_g                       (deslice, weight path)
#   dM     = sum_b dz' z^T ;  dz = M^T dz'      (mix)
#   dU_g   = dz_g / (S_g + eps) ; dS_g = -(dz_g . z_g) / (S_g + eps)
#   dfx_n  = sum_g w_ng dU_g                    (slice, value path)
#   dw^S_ng = f_n . dU_g + dS_g                 (slice, weight path)
#   da_ng  = w_ng (dw_ng - sum_g' w_ng' dw_ng') (softmax Jacobian-vector product)
#   dx_n   = (1/tau) sum_g da_ng W_:g ;  dW = (1/tau) sum_n x_n^T da_n
#   dbeta  = (1/tau) sum_n da_n ; dtau = -(1/tau) sum_{n,g} da_ng a_ng  (App. G.2)
# The split into a deslice part (dw^D) and a slice part (dw^S) is exact because
# da is linear in dw.
# --------------------------------------------------------------------------


def _softmax_vjp(w, dw):
    """da = w * (dw - rowsum(w * dw)): the full softmax Jacobian applied to dw."""
    return w * (dw - (w * dw).sum(axis=1, keepdims=True))


def _param_grads_from_da(x, a, da, W, tau):
    """Gradients of a = (x W + beta)/tau given da (one block of points)."""
    inv = 1.0 / float(tau)
    dx = (da @ _f64(W).T) * inv
    dW = (_f64(x).T @ da) * inv
    db = da.sum(axis=0) * inv
    dtau = -(da * a).sum() * inv
    return dx, dW, db, dtau


def deslice_bwd(x_mid, W_slice, bias, tau, tokens_mixed, dout, heads=None):
    """Gradients of out = w z' w.r.t. z' and, through w, the logit inputs.

    Returns dict: d_tokens_mixed [B,H,G,d], dx_mid [B,N,H,d], dW [H,d,G],
    dbias [H,G], dtau [H] (parameter grads summed over the batch).
    """
    B, N, H, d, G = _shape(x_mid, W_slice)
    dtm = np.full((B, H, G, d), np.nan)
    dx = np.full((B, N, H, d), np.nan)
    dW = np.full((H, d, G), np.nan)
    db = np.full((H, G), np.nan)
    dt = np.full((H,), np.nan)
    for h in _heads(H, heads):
        dW[h] = 0.0
        db[h] = 0.0
        dt[h] = 0.0
        for b in range(B):
            acc = np.zeros((G, d))
            zp = _f64(tokens_mixed[b, h])
            for n0 in range(0, N, _CHUNK):
                n1 = min(N, n0 + _CHUNK)
                x = x_mid[b, n0:n1, h, :]
                a = logits(x, W_slice[h], bias[h], tau[h])
                w, _ = softmax_rows(a)
                dO = _f64(dout[b, n0:n1, h, :])
                acc += w.T @ dO
                dw = dO @ zp.T
                da = _softmax_vjp(w, dw)
                gx, gW, gb, gt = _param_grads_from_da(x, a, da, W_slice[h], tau[h])
                dx[b, n0:n1, h, :] = gx
                dW[h] += gW
                db[h] += gb
                dt[h] += gt
            dtm[b, h] = acc
    return {"d_tokens_mixed": dtm, "dx_mid": dx, "dW": dW, "dbias": db, "dtau": dt}


def mix_bwd(M, tokens, d_tokens_mixed):
    """Backward of z' = M z: dz = M^T dz', dM = sum_b dz' z^T."""
    M = _f64(M)
    dzp = _f64(d_tokens_mixed)
    dz = np.einsum("hgk,bhgc->bhkc", M, dzp)
    dM = np.einsum("bhgc,bhkc->hgk", dzp, _f64(tokens))
    return {"d_tokens": dz, "dM": dM}


def mix_channels(Wc, tokens):
    """Core of the attention-free variant (Sec. 2 after Eq. (1), Sec. 3 variants
    table, "NoTokenAttn"): A is the identity, so the tokens do not interact, and a
    learned linear map acts on the channels of each token, one d x d map per head:
    z'[b,h,g,c] = sum_k Wc[h,c,k] z[b,h,g,k]."""
    return np.einsum("hck,bhgk->bhgc", _f64(Wc), _f64(tokens))


def mix_channels_bwd(Wc, tokens, d_tokens_mixed):
    """Backward of z' = Wc z per token: dz = Wc^T dz', dWc = sum over b and g of dz' z^T."""
    dzp = _f64(d_tokens_mixed)
    dz = np.einsum("hck,bhgc->bhgk", _f64(Wc), dzp)
    dWc = np.einsum("bhgc,bhgk->hck", dzp, _f64(tokens))
    return {"d_tokens": dz, "dWc": dWc}


def slice_bwd(x_mid, fx, W_slice, bias, tau, tokens, wsum, d_tokens, eps=DEFAULT_EPS, heads=None):
    """Gradients of z = U/(S+eps), U = w^T f, S = w^T 1 w.r.t. fx and the logit inputs.

    Returns dict: dx_mid [B,N,H,d], dfx [B,N,H,d], dW [H,d,G], dbias [H,G], dtau [H].
    """
    B, N, H, d, G = _shape(x_mid, W_slice)
    dx = np.full((B, N, H, d), np.nan)
    dfx = np.full((B, N, H, d), np.nan)
    dW = np.full((H, d, G), np.nan)
    db = np.full((H, G), np.nan)
    dt = np.full((H,), np.nan)
    for h in _heads(H, heads):
        dW[h] = 0.0
        db[h] = 0.0
        dt[h] = 0.0
        for b in range(B):
            z = _f64(tokens[b, h])
            dz = _f64(d_tokens[b, h])
            den = _f64(wsum[b, h]) + eps
            dU = dz / den[:, None]
            dS = -(dz * z).sum(axis=1) / den
            for n0 in range(0, N, _CHUNK):
                n1 = min(N, n0 + _CHUNK)
                x = x_mid[b, n0:n1, h, :]
                f = _f64(fx[b, n0:n1, h, :])
                a = logits(x, W_slice[h], bias[h], tau[h])
                w, _ = softmax_rows(a)
                dfx[b, n0:n1, h, :] = w @ dU
                dw = f @ dU.T + dS[None, :]
                da = _softmax_vjp(w, dw)
                gx, gW, gb, gt = _param_grads_from_da(x, a, da, W_slice[h], tau[h])
                dx[b, n0:n1, h, :] = gx
                dW[h] += gW
                db[h] += gb
                dt[h] += gt
    return {"dx_mid": dx, "dfx": dfx, "dW": dW, "dbias": db, "dtau": dt}


def backward(x_mid, fx, W_slice, bias, tau, M, dout, eps=DEFAULT_EPS, heads=None):
    """Full backward of slice -> mix -> deslice given the upstream gradient dout.

    Returns every gradient: dx_mid, dfx, dW, dbias, dtau, dM, plus the token
    gradients d_tokens_mixed and d_tokens.
    """
    fw = forward(x_mid, fx, W_slice, bias, tau, M, eps, heads, points=np.array([], dtype=np.int64))
    dd = deslice_bwd(x_mid, W_slice, bias, tau, fw["tokens_mixed"], dout, heads)
    mb = mix_bwd(M, fw["tokens"], dd["d_tokens_mixed"])
    sb = slice_bwd(x_mid, fx, W_slice, bias, tau, fw["tokens"], fw["wsum"], mb["d_tokens"], eps, heads)
    return {
        "dx_mid": dd["dx_mid"] + sb["dx_mid"],
        "dfx": sb["dfx"],
        "dW": dd["dW"] + sb["dW"],
        "dbias": dd["dbias"] + sb["dbias"],
        "dtau": dd["dtau"] + sb["dtau"],
        "dM": mb["dM"],
        "d_tokens_mixed": dd["d_tokens_mixed"],
        "d_tokens": mb["d_tokens"],
    }
