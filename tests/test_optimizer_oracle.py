"""Pins of the update oracle (``oracle/optimizer.py``): closed forms of the
first and of constant-gradient steps, the decay rules, and agreement with
torch.optim's AdamW and SGD (library routines implementing the same rules)."""
import numpy as np
import pytest

from oracle import optimizer as O


def test_adamw_first_step_closed_form():
    # zero state, t = 1: m_hat = g and v_hat = g^2 exactly, so the step is
    # lr * g / (|g| + eps), plus the decay lr * wd * w
    rng = np.random.default_rng(0)
    w, g = rng.normal(size=50), rng.normal(size=50)
    lr, wd, eps = 1e-3, 0.01, 1e-6
    w1, m1, v1 = O.adamw_step(w, g, 0 * w, 0 * w, 1, lr, 0.9, 0.999, eps, wd)
    expect = w - lr * wd * w - lr * g / (np.abs(g) + eps)
    assert np.allclose(w1, expect, rtol=0, atol=1e-15)
    assert np.allclose(m1, 0.1 * g) and np.allclose(v1, 0.001 * g * g)
    # no decay on biases / LayerNorm parameters
    w1n, _, _ = O.adamw_step(w, g, 0 * w, 0 * w, 1, lr, 0.9, 0.999, eps, wd, decay=False)
    assert np.allclose(w1n, w - lr * g / (np.abs(g) + eps), rtol=0, atol=1e-15)


def test_adamw_constant_gradient():
    # with a constant gradient the bias corrections make m_hat = g and
    # v_hat = g^2 at every step: w_t = w_0 - t * lr * g / (|g| + eps) (no decay)
    g = np.array([0.5, -2.0, 1e-3])
    w = np.zeros(3)
    m, v = np.zeros(3), np.zeros(3)
    for t in range(1, 8):
        w, m, v = O.adamw_step(w, g, m, v, t, 0.1, 0.9, 0.99, 1e-8, 0.0)
    assert np.allclose(w, -7 * 0.1 * g / (np.abs(g) + 1e-8), rtol=1e-12)


def test_sgd_closed_form():
    w, g = np.array([1.0, -2.0]), np.array([0.5, 0.25])
    w1, b1 = O.sgd_step(w, g, np.zeros(2), 1, 0.1, 0.9, 0.0)
    assert np.array_equal(w1, w - 0.1 * g) and np.array_equal(b1, g)
    # second step with the same gradient: b = 0.9 g + g
    w2, b2 = O.sgd_step(w1, g, b1, 2, 0.1, 0.9, 0.0)
    assert np.allclose(w2, w1 - 0.1 * 1.9 * g, rtol=0, atol=1e-15)
    # weight decay enters the gradient
    w3, _ = O.sgd_step(w, g, np.zeros(2), 1, 0.1, 0.9, 0.5)
    assert np.allclose(w3, w - 0.1 * (g + 0.5 * w), rtol=0, atol=1e-15)


def test_against_torch_optim():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(1)
    w0 = rng.normal(size=(6, 5))
    grads = [rng.normal(size=(6, 5)) for _ in range(4)]
    for kind in ("adamw", "sgd"):
        p = torch.nn.Parameter(torch.tensor(w0, dtype=torch.float64))
        if kind == "adamw":
            opt = torch.optim.AdamW([p], lr=1e-2, betas=(0.9, 0.98), eps=1e-6, weight_decay=0.05)
        else:
            opt = torch.optim.SGD([p], lr=1e-2, momentum=0.9, weight_decay=0.05)
        w, m, v, b = w0.copy(), 0 * w0, 0 * w0, 0 * w0
        for t, g in enumerate(grads, start=1):
            p.grad = torch.tensor(g, dtype=torch.float64)
            opt.step()
            if kind == "adamw":
                w, m, v = O.adamw_step(w, g, m, v, t, 1e-2, 0.9, 0.98, 1e-6, 0.05)
            else:
                w, b = O.sgd_step(w, g, b, t, 1e-2, 0.9, 0.05)
        assert np.allclose(p.detach().numpy(), w, rtol=1e-12, atol=1e-14), kind
