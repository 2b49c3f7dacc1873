"""Scalar-loop restatement of the coupling, for tiny inputs only.

TEST INFRASTRUCTURE ONLY (see oracle/__init__.py).  It exists to pin the
vectorised oracle: it uses no numpy contraction at all, only Python floats and
explicit loops over (b, n, h, g, k), and it differentiates by the chain rule
element by element, so a transposed operand or a dropped term in the matrix
formulation of flashslice_oracle.py shows up as a mismatch.

Definitions: paper Sec. 2 ("The Transolver layer") and Appendix G.1; the
temperature gradient as in Appendix G.2.  Inputs are nested Python lists (or
anything indexable) with the shapes documented in flashslice_oracle.py.
"""
from __future__ import annotations

import math


def _weights(x_mid, W, bias, tau, b, n, h, d, G):
    a = []
    for g in range(G):
        s = bias[h][g]
        for k in range(d):
            s += x_mid[b][n][h][k] * W[h][k][g]
        a.append(s / tau[h])
    m = max(a)
    e = [math.exp(v - m) for v in a]
    tot = sum(e)
    return a, [v / tot for v in e]


def forward(x_mid, fx, W, bias, tau, M, eps, B, N, H, d, G):
    """Returns (tokens, wsum, tokens_mixed, out) as nested lists."""
    tokens = [[[[0.0] * d for _ in range(G)] for _ in range(H)] for _ in range(B)]
    wsum = [[[0.0] * G for _ in range(H)] for _ in range(B)]
    for b in range(B):
        for h in range(H):
            U = [[0.0] * d for _ in range(G)]
            S = [0.0] * G
            for n in range(N):
                _, w = _weights(x_mid, W, bias, tau, b, n, h, d, G)
                for g in range(G):
                    S[g] += w[g]
                    for k in range(d):
                        U[g][k] += w[g] * fx[b][n][h][k]
            for g in range(G):
                wsum[b][h][g] = S[g]
                for k in range(d):
                    tokens[b][h][g][k] = U[g][k] / (S[g] + eps)
    tm = [[[[0.0] * d for _ in range(G)] for _ in range(H)] for _ in range(B)]
    for b in range(B):
        for h in range(H):
            for g in range(G):
                for k in range(d):
                    s = 0.0
                    for j in range(G):
                        s += M[h][g][j] * tokens[b][h][j][k]
                    tm[b][h][g][k] = s
    out = [[[[0.0] * d for _ in range(H)] for _ in range(N)] for _ in range(B)]
    for b in range(B):
        for n in range(N):
            for h in range(H):
                _, w = _weights(x_mid, W, bias, tau, b, n, h, d, G)
                for k in range(d):
                    s = 0.0
                    for g in range(G):
                        s += w[g] * tm[b][h][g][k]
                    out[b][n][h][k] = s
    return tokens, wsum, tm, out


def backward(x_mid, fx, W, bias, tau, M, eps, dout, B, N, H, d, G):
    """Returns dict of nested lists: dx_mid, dfx, dW, dbias, dtau, dM."""
    tokens, wsum, tm, _ = forward(x_mid, fx, W, bias, tau, M, eps, B, N, H, d, G)
    dx = [[[[0.0] * d for _ in range(H)] for _ in range(N)] for _ in range(B)]
    dfx = [[[[0.0] * d for _ in range(H)] for _ in range(N)] for _ in range(B)]
    dW = [[[0.0] * G for _ in range(d)] for _ in range(H)]
    db = [[0.0] * G for _ in range(H)]
    dt = [0.0] * H
    dM = [[[0.0] * G for _ in range(G)] for _ in range(H)]
    for b in range(B):
        for h in range(H):
            # deslice: dz'_g = sum_n w_ng dO_n
            dzp = [[0.0] * d for _ in range(G)]
            for n in range(N):
                _, w = _weights(x_mid, W, bias, tau, b, n, h, d, G)
                for g in range(G):
                    for k in range(d):
                        dzp[g][k] += w[g] * dout[b][n][h][k]
            # mix: z' = M z
            dz = [[0.0] * d for _ in range(G)]
            for g in range(G):
                for j in range(G):
                    for k in range(d):
                        dM[h][g][j] += dzp[g][k] * tokens[b][h][j][k]
                        dz[j][k] += M[h][g][j] * dzp[g][k]
            # normalisation z = U / (S + eps)
            dU = [[dz[g][k] / (wsum[b][h][g] + eps) for k in range(d)] for g in range(G)]
            dS = [-sum(dz[g][k] * tokens[b][h][g][k] for k in range(d)) / (wsum[b][h][g] + eps)
                  for g in range(G)]
            for n in range(N):
                a, w = _weights(x_mid, W, bias, tau, b, n, h, d, G)
                # gradient w.r.t. each weight w_ng, from deslice and from slice
                dw = []
                for g in range(G):
                    s = dS[g]
                    for k in range(d):
                        s += dout[b][n][h][k] * tm[b][h][g][k]
                        s += fx[b][n][h][k] * dU[g][k]
                    dw.append(s)
                for k in range(d):
                    dfx[b][n][h][k] = sum(w[g] * dU[g][k] for g in range(G))
                # softmax: da_g = sum_j (dw_j) * dw_j/da_g, dw_j/da_g = w_j (delta_jg - w_g)
                for g in range(G):
                    da = 0.0
                    for j in range(G):
                        jac = w[j] * ((1.0 if j == g else 0.0) - w[g])
                        da += dw[j] * jac
                    # a_g = (sum_k x_k W_kg + beta_g) / tau
                    for k in range(d):
                        dx[b][n][h][k] += da * W[h][k][g] / tau[h]
                        dW[h][k][g] += da * x_mid[b][n][h][k] / tau[h]
                    db[h][g] += da / tau[h]
                    dt[h] += -da * a[g] / tau[h]
    return {"dx_mid": dx, "dfx": dfx, "dW": dW, "dbias": db, "dtau": dt, "dM": dM}


def mix_channels(Wc, tokens, B, H, G, d):
    """z'[b][h][g][c] = sum_k Wc[h][c][k] z[b][h][g][k], by loops (the NoTokenAttn
    core: a per-token channel map, Sec. 2 after Eq. (1))."""
    out = [[[[0.0] * d for _ in range(G)] for _ in range(H)] for _ in range(B)]
    for b in range(B):
        for h in range(H):
            for g in range(G):
                for c in range(d):
                    acc = 0.0
                    for k in range(d):
                        acc += Wc[h][c][k] * tokens[b][h][g][k]
                    out[b][h][g][c] = acc
    return out


def mix_channels_bwd(Wc, tokens, d_tokens_mixed, B, H, G, d):
    """Chain rule of mix_channels element by element: (d_tokens, dWc)."""
    dz = [[[[0.0] * d for _ in range(G)] for _ in range(H)] for _ in range(B)]
    dWc = [[[0.0] * d for _ in range(d)] for _ in range(H)]
    for b in range(B):
        for h in range(H):
            for g in range(G):
                for c in range(d):
                    up = d_tokens_mixed[b][h][g][c]
                    for k in range(d):
                        dz[b][h][g][k] += Wc[h][c][k] * up
                        dWc[h][c][k] += up * tokens[b][h][g][k]
    return dz, dWc
