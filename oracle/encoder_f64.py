"""Float64 CPU oracle of a slice of post-LN BERT encoder layers, forward and backward.

TEST INFRASTRUCTURE ONLY.  Nothing in the library's product path imports,
links or calls this module; only the tests, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` do.  It shares no code with the CUDA path.

What it computes (the plain definition, written out in float64):

* Encoder layer = self-attention block, intermediate block and output block,
  each ending in a linear layer, the attention and output blocks with a
  residual connection (Sec. II-C).  Post-LayerNorm placement and the GELU
  intermediate activation follow BERT, which the paper builds on (Sec. II-C).
* Q, K, V are the input times three ``(h, v)`` matrices (Sec. II-C); here
  ``v = h = A * D`` and the three are stacked as ``Wqkv[3H, H]`` (rows Q | K | V,
  head-major inside each block).
* Attention(Q, K, V) = softmax(Q K^T / sqrt(d_k)) V per head (Eq. 1), with
  ``d_k = D`` the per-head key width, over the valid keys ``j < len_b`` only
  (key-padding mask: padded keys get probability exactly 0).  All S query rows
  are computed, padded ones included.
* Backward: every activation and parameter gradient of the slice, layers in
  reverse order (Sec. III: gradients are computed in the reverse order of the
  forward pass and used locally).  The attention backward uses the explicit
  ``sum_k P_ik dP_ik`` term, not the ``rowsum(dO * O)`` shortcut.

Conventions: ``Linear(x) = x W^T + b`` with ``W[out, in]``; LayerNorm uses the
biased (divide-by-H) variance and ``rstd = 1 / sqrt(var + eps)``; GELU is the
exact ``z * Phi(z)`` with the error function from ``scipy.special`` (a library
routine).  Matrix products use numpy ``@`` as a library primitive; there is no
blocking, fusion or reordering beyond the definition.
"""
from __future__ import annotations

import math

import numpy as np
from scipy.special import erf

PARAM_NAMES = (
    "Wqkv", "bqkv", "Wo", "bo", "gamma1", "beta1",
    "W1", "b1", "W2", "b2", "gamma2", "beta2",
)


def gelu(z):
    """GELU(z) = z * Phi(z), Phi the standard normal CDF (BERT's exact form)."""
    return z * 0.5 * (1.0 + erf(z / math.sqrt(2.0)))


def gelu_grad(z):
    """d/dz [z Phi(z)] = Phi(z) + z phi(z), phi the standard normal density."""
    Phi = 0.5 * (1.0 + erf(z / math.sqrt(2.0)))
    phi = np.exp(-0.5 * z * z) / math.sqrt(2.0 * math.pi)
    return Phi + z * phi


def layer_norm(U, gamma, beta, eps):
    """Row LayerNorm of U[T, H]; returns (Y, xhat, rstd)."""
    mu = U.mean(axis=1, keepdims=True)
    var = ((U - mu) ** 2).mean(axis=1, keepdims=True)
    rstd = 1.0 / np.sqrt(var + eps)
    xhat = (U - mu) * rstd
    return gamma * xhat + beta, xhat, rstd


def layer_norm_backward(dY, xhat, rstd, gamma):
    """Gradient of Y = gamma * xhat + beta w.r.t. U, gamma and beta."""
    h = dY * gamma
    dU = rstd * (h - h.mean(axis=1, keepdims=True)
                 - xhat * (h * xhat).mean(axis=1, keepdims=True))
    return dU, (dY * xhat).sum(axis=0), dY.sum(axis=0)


def attention_forward(Q, K, V, lens):
    """Masked scaled dot-product attention (Eq. 1) per sequence and head.

    Q, K, V: [B, S, A, D].  Returns ctx [B, S, A, D] and the probabilities
    P [B, A, S, S] (zero in the masked key columns).
    """
    B, S, A, D = Q.shape
    ctx = np.zeros_like(Q)
    P = np.zeros((B, A, S, S))
    for b in range(B):
        n = int(lens[b])
        for a in range(A):
            s = Q[b, :, a, :] @ K[b, :n, a, :].T / math.sqrt(D)
            e = np.exp(s - s.max(axis=1, keepdims=True))
            p = e / e.sum(axis=1, keepdims=True)
            P[b, a, :, :n] = p
            ctx[b, :, a, :] = p @ V[b, :n, a, :]
    return ctx, P


def attention_backward(dctx, Q, K, V, P, lens):
    """Gradients of Eq. 1 w.r.t. Q, K, V given dctx, all [B, S, A, D]."""
    B, S, A, D = Q.shape
    dQ, dK, dV = np.zeros_like(Q), np.zeros_like(K), np.zeros_like(V)
    for b in range(B):
        n = int(lens[b])
        for a in range(A):
            p = P[b, a, :, :n]
            dO = dctx[b, :, a, :]
            dV[b, :n, a, :] = p.T @ dO
            dP = dO @ V[b, :n, a, :].T
            dS = p * (dP - (p * dP).sum(axis=1, keepdims=True))
            dQ[b, :, a, :] = dS @ K[b, :n, a, :] / math.sqrt(D)
            dK[b, :n, a, :] = dS.T @ Q[b, :, a, :] / math.sqrt(D)
    return dQ, dK, dV


def layer_forward(X, lens, p, heads, eps):
    """One post-LN encoder layer.  X [B, S, H] -> Y [B, S, H] and a cache."""
    B, S, H = X.shape
    D = H // heads
    f = lambda t: np.asarray(t, dtype=np.float64)
    p = {k: f(v) for k, v in p.items()}
    Xf = f(X).reshape(B * S, H)
    QKV = Xf @ p["Wqkv"].T + p["bqkv"]
    Q = QKV[:, :H].reshape(B, S, heads, D)
    K = QKV[:, H:2 * H].reshape(B, S, heads, D)
    V = QKV[:, 2 * H:].reshape(B, S, heads, D)
    ctx4, P = attention_forward(Q, K, V, lens)
    ctx = ctx4.reshape(B * S, H)
    U1 = ctx @ p["Wo"].T + p["bo"] + Xf
    X1, xhat1, rstd1 = layer_norm(U1, p["gamma1"], p["beta1"], eps)
    Z = X1 @ p["W1"].T + p["b1"]
    G = gelu(Z)
    U2 = G @ p["W2"].T + p["b2"] + X1
    Y, xhat2, rstd2 = layer_norm(U2, p["gamma2"], p["beta2"], eps)
    cache = dict(X=Xf, Q=Q, K=K, V=V, P=P, ctx=ctx, xhat1=xhat1, rstd1=rstd1, X1=X1,
                 Z=Z, G=G, xhat2=xhat2, rstd2=rstd2, lens=np.asarray(lens), p=p,
                 shape=(B, S, H), heads=heads)
    return Y.reshape(B, S, H), cache


def layer_backward(dY, cache):
    """Backward of ``layer_forward``: returns dX [B, S, H] and the 12 gradients."""
    B, S, H = cache["shape"]
    p = cache["p"]
    dYf = np.asarray(dY, dtype=np.float64).reshape(B * S, H)
    dU2, dgamma2, dbeta2 = layer_norm_backward(dYf, cache["xhat2"], cache["rstd2"], p["gamma2"])
    db2 = dU2.sum(axis=0)
    dW2 = dU2.T @ cache["G"]
    dG = dU2 @ p["W2"]
    dZ = dG * gelu_grad(cache["Z"])
    db1 = dZ.sum(axis=0)
    dW1 = dZ.T @ cache["X1"]
    dX1 = dZ @ p["W1"] + dU2
    dU1, dgamma1, dbeta1 = layer_norm_backward(dX1, cache["xhat1"], cache["rstd1"], p["gamma1"])
    dbo = dU1.sum(axis=0)
    dWo = dU1.T @ cache["ctx"]
    dctx = (dU1 @ p["Wo"]).reshape(cache["Q"].shape)
    dQ, dK, dV = attention_backward(dctx, cache["Q"], cache["K"], cache["V"], cache["P"],
                                    cache["lens"])
    dQKV = np.concatenate([dQ.reshape(B * S, H), dK.reshape(B * S, H),
                           dV.reshape(B * S, H)], axis=1)
    dbqkv = dQKV.sum(axis=0)
    dWqkv = dQKV.T @ cache["X"]
    dX = dQKV @ p["Wqkv"] + dU1
    grads = dict(Wqkv=dWqkv, bqkv=dbqkv, Wo=dWo, bo=dbo, gamma1=dgamma1, beta1=dbeta1,
                 W1=dW1, b1=db1, W2=dW2, b2=db2, gamma2=dgamma2, beta2=dbeta2)
    return dX.reshape(B, S, H), grads


def slice_forward(X, lens, params, heads, eps):
    """Forward over a contiguous slice: layer l's output is layer l+1's input."""
    caches = []
    for p in params:
        X, c = layer_forward(X, lens, p, heads, eps)
        caches.append(c)
    return X, caches


def slice_backward(dY, caches):
    """Backward over the slice in reverse layer order; returns dX and per-layer grads."""
    grads = [None] * len(caches)
    for i in range(len(caches) - 1, -1, -1):
        dY, grads[i] = layer_backward(dY, caches[i])
    return dY, grads


def slice_step(X, lens, dY, params, heads, eps):
    """Forward then backward of the slice; returns (Y, dX, grads)."""
    Y, caches = slice_forward(X, lens, params, heads, eps)
    dX, grads = slice_backward(dY, caches)
    return Y, dX, grads
