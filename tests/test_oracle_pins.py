"""Pins of the float64 oracle against facts the paper and mathematics fix.

Each check below is written so that a plausible slip in the oracle (a dropped
term, a wrong sign, index or scale, a transposed operand) makes at least one
of them fail; ``test_planted_mistakes_are_caught`` plants such slips in a copy
of the oracle and asserts exactly that.  No GPU is needed.
"""
import importlib.util
import math
import os

import numpy as np
import pytest

from oracle import encoder_f64 as ORC
from paper_2202_11836_gb300 import synth

HERE = os.path.dirname(os.path.abspath(__file__))
ORACLE_SRC = os.path.join(os.path.dirname(HERE), "oracle", "encoder_f64.py")


# --------------------------------------------------------------------------
# small helpers (inputs only; no encoder arithmetic)
# --------------------------------------------------------------------------
def tiny_case(B=2, S=7, H=8, A=2, F=12, seed=5, lens=(7, 4)):
    g = np.random.default_rng(seed)
    X = g.normal(0, 1, (B, S, H))
    p = {
        "Wqkv": g.normal(0, 0.3, (3 * H, H)), "bqkv": g.normal(0, 0.1, 3 * H),
        "Wo": g.normal(0, 0.3, (H, H)), "bo": g.normal(0, 0.1, H),
        "gamma1": 1 + g.normal(0, 0.1, H), "beta1": g.normal(0, 0.1, H),
        "W1": g.normal(0, 0.3, (F, H)), "b1": g.normal(0, 0.1, F),
        "W2": g.normal(0, 0.3, (H, F)), "b2": g.normal(0, 0.1, H),
        "gamma2": 1 + g.normal(0, 0.1, H), "beta2": g.normal(0, 0.1, H),
    }
    return X, np.array(lens, dtype=np.int32), p, A


def tiny_fp32_workload_inputs(layers=2):
    w = synth.WORKLOADS["tiny-fp32"]
    params = [synth.layer_params(l, w.hidden, w.ffn, "fp32", affine="random")
              for l in range(layers)]
    return w, synth.activations(w).astype(np.float64), synth.lengths(w), params


# --------------------------------------------------------------------------
# checks (take the oracle module so that planted mistakes can be fed in)
# --------------------------------------------------------------------------
def check_gelu_table(orc):
    rows = [l.split() for l in open(os.path.join(HERE, "golden", "normal_cdf.txt"))
            if l.strip() and not l.startswith("#")]
    for z, phi in rows:
        z, phi = float(z), float(phi)
        assert abs(orc.gelu(np.array(z)) - z * phi) <= 1e-14, (z, phi)
    assert orc.gelu(np.array(0.0)) == 0.0
    assert abs(orc.gelu_grad(np.array(0.0)) - 0.5) <= 1e-15
    # derivative: Phi(1) + phi(1) with phi(1) = exp(-1/2)/sqrt(2 pi)
    assert abs(orc.gelu_grad(np.array(1.0)) - (0.841344746068543 + 0.241970724519143)) <= 1e-13


def check_softmax_rows(orc):
    X, lens, p, A = tiny_case()
    _, c = orc.layer_forward(X, lens, p, A, 1e-12)
    P = c["P"]
    for b, n in enumerate(lens):
        assert np.all(P[b, :, :, n:] == 0.0)
        assert np.max(np.abs(P[b, :, :, :n].sum(-1) - 1.0)) <= 1e-14
        assert np.all(P[b, :, :, :n] > 0)


def check_attention_closed_forms(orc):
    # Scores Q.K/sqrt(D) of ln 3 and 0 give probabilities 3/4 and 1/4.
    D = 64
    Q = np.zeros((1, 2, 1, D)); K = np.zeros((1, 2, 1, D)); V = np.zeros((1, 2, 1, D))
    Q[0, :, 0, 0] = 1.0
    K[0, 0, 0, 0] = math.sqrt(D) * math.log(3.0)
    V[0, 0, 0, 1] = 1.0; V[0, 1, 0, 2] = 1.0
    ctx, P = orc.attention_forward(Q, K, V, np.array([2]))
    assert abs(P[0, 0, 0, 0] - 0.75) <= 1e-15 and abs(P[0, 0, 0, 1] - 0.25) <= 1e-15
    assert abs(ctx[0, 1, 0, 1] - 0.75) <= 1e-15 and abs(ctx[0, 1, 0, 2] - 0.25) <= 1e-15
    # Zero queries give uniform attention: ctx_i = mean of the valid V rows.
    g = np.random.default_rng(1)
    B, S, A, D = 2, 6, 2, 4
    Q = np.zeros((B, S, A, D)); K = g.normal(size=(B, S, A, D)); V = g.normal(size=(B, S, A, D))
    lens = np.array([6, 3])
    ctx, _ = orc.attention_forward(Q, K, V, lens)
    for b, n in enumerate(lens):
        np.testing.assert_allclose(ctx[b], np.broadcast_to(V[b, :n].mean(0), (S, A, D)),
                                   rtol=0, atol=1e-14)
    # A single valid key: every query returns V_0.
    Q = g.normal(size=(B, S, A, D))
    ctx, _ = orc.attention_forward(Q, K, V, np.array([1, 1]))
    for b in range(B):
        np.testing.assert_allclose(ctx[b], np.broadcast_to(V[b, 0], (S, A, D)), rtol=0, atol=1e-15)


def check_layernorm_moments(orc):
    g = np.random.default_rng(2)
    U = g.normal(3.0, 2.0, (9, 16))
    for eps in (1e-12, 0.5):
        Y, xhat, rstd = orc.layer_norm(U, np.ones(16), np.zeros(16), eps)
        var = ((U - U.mean(1, keepdims=True)) ** 2).sum(1) / 16
        assert np.max(np.abs(xhat.mean(1))) <= 1e-13
        np.testing.assert_allclose((xhat ** 2).mean(1), var / (var + eps), rtol=0, atol=1e-13)
    gam, bet = g.normal(size=16), g.normal(size=16)
    Y, xhat, _ = orc.layer_norm(U, gam, bet, 1e-12)
    np.testing.assert_allclose(Y, gam * xhat + bet, rtol=0, atol=1e-14)


def check_post_ln_output(orc):
    # Post-LN: with gamma 1, beta 0 the layer output rows are normalised.
    w, X, lens, _ = tiny_fp32_workload_inputs(1)
    p = synth.layer_params(0, w.hidden, w.ffn, "fp32", affine="bert")
    Y, _ = orc.layer_forward(X, lens, p, w.heads, 1e-12)
    Y = Y.reshape(-1, w.hidden)
    assert np.max(np.abs(Y.mean(1))) <= 1e-12
    assert np.max(np.abs((Y ** 2).mean(1) - 1.0)) <= 1e-9


def brute_force_layer(X, lens, p, A, eps):
    """Encoder layer with scalar loops only (independent of the oracle's code)."""
    B, S, H = X.shape
    D = H // A
    F = len(p["b1"])

    def lin(x, W, b):
        return [sum(W[o][i] * x[i] for i in range(len(x))) + b[o] for o in range(len(b))]

    def ln(u, g, be):
        mu = sum(u) / len(u)
        var = sum((v - mu) ** 2 for v in u) / len(u)
        return [g[k] * (u[k] - mu) / math.sqrt(var + eps) + be[k] for k in range(len(u))]

    Y = np.zeros((B, S, H))
    for b in range(B):
        qkv = [lin(list(X[b, s]), p["Wqkv"], p["bqkv"]) for s in range(S)]
        n = int(lens[b])
        for i in range(S):
            ctx = [0.0] * H
            for a in range(A):
                sc = []
                for j in range(n):
                    sc.append(sum(qkv[i][a * D + d] * qkv[j][H + a * D + d] for d in range(D))
                              / math.sqrt(D))
                mx = max(sc)
                ex = [math.exp(v - mx) for v in sc]
                tot = sum(ex)
                for d in range(D):
                    ctx[a * D + d] = sum(ex[j] / tot * qkv[j][2 * H + a * D + d] for j in range(n))
            ao = lin(ctx, p["Wo"], p["bo"])
            x1 = ln([ao[k] + X[b, i, k] for k in range(H)], p["gamma1"], p["beta1"])
            z = lin(x1, p["W1"], p["b1"])
            gz = [v * 0.5 * (1 + math.erf(v / math.sqrt(2))) for v in z]
            o = lin(gz, p["W2"], p["b2"])
            Y[b, i] = ln([o[k] + x1[k] for k in range(H)], p["gamma2"], p["beta2"])
    assert F == len(p["W1"])
    return Y


def check_brute_force(orc):
    X, lens, p, A = tiny_case()
    Y, _ = orc.layer_forward(X, lens, p, A, 1e-5)
    Yb = brute_force_layer(X, lens, p, A, 1e-5)
    np.testing.assert_allclose(Y, Yb, rtol=0, atol=1e-12)


def check_mask_equals_truncation(orc):
    X, lens, p, A = tiny_case(B=1, S=9, lens=(5,))
    params = [p, tiny_case(seed=9)[2]]
    Y, caches = orc.slice_forward(X, lens, params, A, 1e-12)
    Yt, caches_t = orc.slice_forward(X[:, :5], np.array([5]), params, A, 1e-12)
    np.testing.assert_allclose(Y[:, :5], Yt, rtol=0, atol=1e-13)
    # Perturbing padded rows leaves the valid rows unchanged.
    X2 = X.copy(); X2[:, 5:] += 3.0
    Y2, _ = orc.slice_forward(X2, lens, params, A, 1e-12)
    np.testing.assert_allclose(Y2[:, :5], Y[:, :5], rtol=0, atol=1e-13)
    # With the upstream gradient zero on padded rows, every weight gradient equals
    # the truncated run's and dX is exactly zero on padded rows.
    g = np.random.default_rng(3)
    dY = g.normal(size=Y.shape); dY[:, 5:] = 0.0
    dX, grads = orc.slice_backward(dY, caches)
    dXt, grads_t = orc.slice_backward(dY[:, :5], caches_t)
    assert np.all(dX[:, 5:] == 0.0)
    np.testing.assert_allclose(dX[:, :5], dXt, rtol=0, atol=1e-13)
    for gl, gt in zip(grads, grads_t):
        for k in ORC.PARAM_NAMES:
            np.testing.assert_allclose(gl[k], gt[k], rtol=0, atol=1e-12 * (1 + np.abs(gt[k]).max()))


def check_identity_layer(orc):
    """Closed form of a layer that is the identity map.

    eps = 0, input rows with mean 0 and variance 1, all weights and biases zero
    except Wo = I and gamma = 1: attention gives ctx = 0 (V = 0), so U1 = X,
    X1 = LN(X) = X, G = GELU(0) = 0 and Y = LN(X1) = X.  The gradients then
    have closed forms: with J = I - (1 1^T + x x^T)/H per row, dU = J dY is the
    gradient at both LayerNorms, dX = dU, dV_j = (1/len) sum_i dU_i for valid
    keys, dQ = dK = 0, and every weight gradient is the outer product of the
    output gradient with the layer input (dW = dy^T x) or zero.
    """
    B, S, H, A, F = 2, 6, 8, 2, 12
    D = H // A
    g = np.random.default_rng(4)
    X = g.normal(size=(B, S, H))
    X = X - X.mean(-1, keepdims=True)
    X = X / np.sqrt((X ** 2).mean(-1, keepdims=True))
    lens = np.array([6, 4])
    p = {k: np.zeros_like(v) for k, v in tiny_case(B, S, H, A, F)[2].items()}
    p["Wo"] = np.eye(H); p["gamma1"] = np.ones(H); p["gamma2"] = np.ones(H)
    Y, caches = orc.slice_forward(X, lens, [p], A, 0.0)
    np.testing.assert_allclose(Y, X, rtol=0, atol=1e-13)
    dY = g.normal(size=(B, S, H))
    dX, (gr,) = orc.slice_backward(dY, caches)
    dU = dY - dY.mean(-1, keepdims=True) - X * (dY * X).mean(-1, keepdims=True)
    tol = dict(rtol=0, atol=1e-12)
    np.testing.assert_allclose(dX, dU, **tol)
    for k in ("W1", "b1", "W2", "Wo"):
        assert np.all(gr[k] == 0.0), k
    col = lambda t: t.reshape(-1, H).sum(0)
    np.testing.assert_allclose(gr["beta2"], col(dY), **tol)
    np.testing.assert_allclose(gr["gamma2"], col(dY * X), **tol)
    np.testing.assert_allclose(gr["b2"], col(dU), **tol)
    np.testing.assert_allclose(gr["beta1"], col(dU), **tol)
    np.testing.assert_allclose(gr["gamma1"], col(dU * X), **tol)
    np.testing.assert_allclose(gr["bo"], col(dU), **tol)
    dV = np.zeros((B, S, H))
    for b, n in enumerate(lens):
        dV[b, :n] = dU[b].sum(0) / n
    np.testing.assert_allclose(gr["bqkv"][:2 * H], 0.0, **tol)
    np.testing.assert_allclose(gr["bqkv"][2 * H:], col(dV), **tol)
    np.testing.assert_allclose(gr["Wqkv"][:2 * H], 0.0, **tol)
    np.testing.assert_allclose(gr["Wqkv"][2 * H:], dV.reshape(-1, H).T @ X.reshape(-1, H), **tol)
    assert D == 4


def check_uniform_attention_wo_grad(orc):
    """Q = K = 0 and V rows all equal v: every ctx row is v, so dWo = outer(dbo, v)."""
    X, lens, p, A = tiny_case()
    H = X.shape[-1]
    p = dict(p)
    p["Wqkv"] = p["Wqkv"].copy(); p["Wqkv"][:] = 0.0
    v = np.random.default_rng(7).normal(size=H)
    p["bqkv"] = np.concatenate([np.zeros(2 * H), v])
    Y, caches = orc.slice_forward(X, lens, [p], A, 1e-12)
    dX, (gr,) = orc.slice_backward(np.random.default_rng(8).normal(size=Y.shape), caches)
    np.testing.assert_allclose(gr["Wo"], np.outer(gr["bo"], v), rtol=0, atol=1e-12)


def finite_difference_errors(orc, n_per_tensor=6, seed=11):
    """Central differences of L = sum(Y * Gup) vs the analytic gradients."""
    w, X, lens, params = tiny_fp32_workload_inputs(2)
    X = X[:2, :20]
    lens = np.array([20, 13], dtype=np.int32)
    params = [{k: v.astype(np.float64) for k, v in p.items()} for p in params]
    g = np.random.default_rng(seed)
    Gup = g.normal(size=X.shape)
    eps = 1e-12

    def loss():
        Y, _ = orc.slice_forward(X, lens, params, w.heads, eps)
        return float((Y * Gup).sum())

    _, caches = orc.slice_forward(X, lens, params, w.heads, eps)
    dX, grads = orc.slice_backward(Gup, caches)
    worst = 0.0

    def probe(arr, idx, analytic, scale):
        nonlocal worst
        old = arr[idx]
        h = 1e-6 * max(1.0, abs(old))
        arr[idx] = old + h; lp = loss()
        arr[idx] = old - h; lm = loss()
        arr[idx] = old
        fd = (lp - lm) / (2 * h)
        worst = max(worst, abs(fd - analytic) / max(abs(analytic), scale))

    # input rows at the mask boundary and elsewhere
    for b, n in enumerate(lens):
        for s in {0, int(n) - 1, min(int(n), X.shape[1] - 1), X.shape[1] - 1}:
            for hcol in g.choice(X.shape[2], 2, replace=False):
                probe(X, (b, s, hcol), dX[b, s, hcol], np.abs(dX).max())
    for li, p in enumerate(params):
        for k in ORC.PARAM_NAMES:
            for _ in range(n_per_tensor):
                idx = tuple(int(g.integers(0, d)) for d in p[k].shape)
                probe(p[k], idx, grads[li][k][idx], np.abs(grads[li][k]).max())
    return worst


def check_finite_differences(orc):
    assert finite_difference_errors(orc, n_per_tensor=3) <= 1e-6


def check_batch_permutation(orc):
    X, lens, p, A = tiny_case(B=3, lens=(7, 2, 5))
    perm = np.array([2, 0, 1])
    Y, c = orc.slice_forward(X, lens, [p], A, 1e-12)
    Yp, cp = orc.slice_forward(X[perm], lens[perm], [p], A, 1e-12)
    np.testing.assert_allclose(Yp, Y[perm], rtol=0, atol=1e-14)


def check_slice_composition(orc):
    X, lens, p, A = tiny_case()
    q = tiny_case(seed=19)[2]
    Y, c = orc.slice_forward(X, lens, [p, q], A, 1e-12)
    Y1, c1 = orc.slice_forward(X, lens, [p], A, 1e-12)
    Y2, c2 = orc.slice_forward(Y1, lens, [q], A, 1e-12)
    np.testing.assert_array_equal(Y, Y2)
    dY = np.random.default_rng(0).normal(size=Y.shape)
    dM, g2 = orc.slice_backward(dY, c2)
    dX, g1 = orc.slice_backward(dM, c1)
    dXf, gf = orc.slice_backward(dY, c)
    np.testing.assert_array_equal(dX, dXf)


ALL_CHECKS = [check_gelu_table, check_softmax_rows, check_attention_closed_forms,
              check_layernorm_moments, check_post_ln_output, check_brute_force,
              check_mask_equals_truncation, check_identity_layer,
              check_uniform_attention_wo_grad, check_finite_differences,
              check_batch_permutation, check_slice_composition]


@pytest.mark.parametrize("check", ALL_CHECKS, ids=lambda f: f.__name__)
def test_oracle_pin(check):
    check(ORC)


def test_finite_differences_dense():
    """All 12 parameter tensors of both layers, 8 entries each, plus boundary input rows."""
    assert finite_difference_errors(ORC, n_per_tensor=8, seed=23) <= 1e-6


# --------------------------------------------------------------------------
# planted mistakes: each must be caught by at least one check
# --------------------------------------------------------------------------
MUTATIONS = {
    "scale_1_over_D": ("/ math.sqrt(D)\n            e", "/ D\n            e"),
    "eps_outside_sqrt": ("np.sqrt(var + eps)", "(np.sqrt(var) + eps)"),
    "unbiased_variance": ("var = ((U - mu) ** 2).mean(axis=1, keepdims=True)",
                          "var = ((U - mu) ** 2).sum(axis=1, keepdims=True) / (U.shape[1] - 1)"),
    "gelu_wrong_cdf": ("z * 0.5 * (1.0 + erf(z / math.sqrt(2.0)))", "z * 0.5 * (1.0 + erf(z / 2.0))"),
    "gelu_grad_missing_term": ("return Phi + z * phi", "return Phi"),
    "no_attention_residual": ('+ p["bo"] + Xf', '+ p["bo"]'),
    "no_ffn_residual_grad": ('dX1 = dZ @ p["W1"] + dU2', 'dX1 = dZ @ p["W1"]'),
    "softmax_grad_no_rowdot": ("dS = p * (dP - (p * dP).sum(axis=1, keepdims=True))", "dS = p * dP"),
    "dK_missing_scale": ("dK[b, :n, a, :] = dS.T @ Q[b, :, a, :] / math.sqrt(D)",
                         "dK[b, :n, a, :] = dS.T @ Q[b, :, a, :]"),
    "ln_grad_sign": ("- xhat * (h * xhat).mean", "+ xhat * (h * xhat).mean"),
    "wo_grad_transposed": ('dWo = dU1.T @ cache["ctx"]', 'dWo = (cache["ctx"].T @ dU1)'),
    "v_grad_unmasked": ("dV[b, :n, a, :] = p.T @ dO", "dV[b, :n, a, :] = p.T @ dO * (n / S)"),
    "dgamma_from_dU": ("(dY * xhat).sum(axis=0), dY.sum(axis=0)", "(dU * xhat).sum(axis=0), dY.sum(axis=0)"),
}


def load_mutant(old, new):
    src = open(ORACLE_SRC).read()
    assert src.count(old) >= 1, old
    src = src.replace(old, new, 1)
    spec = importlib.util.spec_from_loader("oracle_mutant", loader=None)
    mod = importlib.util.module_from_spec(spec)
    exec(compile(src, "oracle_mutant", "exec"), mod.__dict__)
    return mod


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_planted_mistakes_are_caught(name):
    mutant = load_mutant(*MUTATIONS[name])
    caught = []
    for check in ALL_CHECKS:
        try:
            check(mutant)
        except (AssertionError, ValueError, IndexError):
            caught.append(check.__name__)
    assert caught, f"planted mistake {name} passed every pin"
