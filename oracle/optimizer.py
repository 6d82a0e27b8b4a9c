"""Float64 oracle of the local parameter update of a slice (Sec. III).

TEST INFRASTRUCTURE ONLY.  Nothing in the library's product path imports,
links or calls this module; only the tests do.  It shares no code with the
CUDA update kernel (``csrc/optimizer.cu``).

After its backward pass every device updates the weights of its own layers
with the gradients it computed, without sending them anywhere (Sec. III).
The paper does not name the optimizer; BERT, which it trains, uses Adam with
decoupled weight decay on the weight matrices.  Two rules are provided:

* ``adamw_step``: Adam (Kingma & Ba, Algorithm 1: first and second moment
  estimates with bias correction) with decoupled weight decay (Loshchilov &
  Hutter): ``w <- w - lr * wd * w`` (decay, weight matrices only) and
  ``w <- w - lr * m_hat / (sqrt(v_hat) + eps)``.
* ``sgd_step``: SGD with heavy-ball momentum, weight decay added to the
  gradient: ``b <- mu * b + (g + wd * w)``, ``w <- w - lr * b`` (first step:
  ``b = g + wd * w``).

Readings: weight decay applies to the four weight matrices (``Wqkv``, ``Wo``,
``W1``, ``W2``) and not to biases or LayerNorm parameters (BERT's choice); the
update runs on fp32 master weights, and a bf16 slice's parameters are the
master weights rounded to bf16 (round to nearest even) after every step.
"""
from __future__ import annotations

import numpy as np

DECAYED = ("Wqkv", "Wo", "W1", "W2")


def adamw_step(w, g, m, v, t, lr, beta1, beta2, eps, wd, decay=True):
    """One AdamW step (t = 1 for the first); returns new (w, m, v) in float64."""
    w, g, m, v = (np.asarray(a, np.float64) for a in (w, g, m, v))
    m = beta1 * m + (1.0 - beta1) * g
    v = beta2 * v + (1.0 - beta2) * g * g
    m_hat = m / (1.0 - beta1 ** t)
    v_hat = v / (1.0 - beta2 ** t)
    if decay:
        w = w - lr * wd * w
    w = w - lr * m_hat / (np.sqrt(v_hat) + eps)
    return w, m, v


def sgd_step(w, g, b, t, lr, momentum, wd, decay=True):
    """One SGD-with-momentum step; returns new (w, b) in float64."""
    w, g, b = (np.asarray(a, np.float64) for a in (w, g, b))
    d = g + (wd * w if decay else 0.0)
    b = d if t == 1 else momentum * b + d
    return w - lr * b, b
