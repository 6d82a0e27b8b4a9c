"""Shared helpers of the GPU parity tests: tolerance metrics and a runner that
executes one slice on the GPU through the C ABI and the float64 oracle on the
same seeded inputs.

Tolerances (the spec bars): fp32 slices maxrel <= 1e-4; bf16 slices
maxrel <= 2e-2 and l2rel <= 5e-3, per output tensor, where
    maxrel = max_i |g_i - o_i| / max_i |o_i|,   l2rel = ||g - o||_2 / ||o||_2.
"""
from __future__ import annotations

import numpy as np

from oracle import encoder_f64 as ORC
from paper_2202_11836_gb300 import synth

TOL = {"fp32": dict(maxrel=1e-4, l2rel=1e-4), "bf16": dict(maxrel=2e-2, l2rel=5e-3)}


def maxrel(g, o):
    g = np.asarray(g, np.float64); o = np.asarray(o, np.float64)
    den = np.abs(o).max()
    return float(np.abs(g - o).max() / den) if den > 0 else float(np.abs(g).max())


def l2rel(g, o):
    g = np.asarray(g, np.float64); o = np.asarray(o, np.float64)
    den = np.linalg.norm(o)
    return float(np.linalg.norm(g - o) / den) if den > 0 else float(np.linalg.norm(g))


def assert_close(name, g, o, dtype):
    t = TOL[dtype]
    mr, lr = maxrel(g, o), l2rel(g, o)
    assert mr <= t["maxrel"] and lr <= t["l2rel"], f"{name}: maxrel {mr:.3e} l2rel {lr:.3e} ({dtype})"
    return mr, lr


def to_device(a, dtype):
    import torch
    t = torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).cuda()
    return t.to(torch.bfloat16) if dtype == "bf16" else t


def to_host(t):
    return t.float().cpu().numpy().astype(np.float64)


def run_gpu_slice(w, X, lens, dY, params, affine_layers, eps=1e-12, steps=1, profiling=False,
                  graph=False):
    """Runs forward+backward of workload ``w`` on the GPU; returns (Y, dX, grads).

    ``steps`` > 1 repeats the step back to back on one stream (results of the
    last one are returned); ``profiling`` runs every kernel in line on the
    caller's stream (per-kernel timing mode); ``graph`` captures the step as
    the benchmark runs it (sky_slice_step_graph_create) and returns the
    results of a replay into zeroed outputs."""
    import torch
    from paper_2202_11836_gb300.slice import EncoderSlice
    B = X.shape[0]
    with EncoderSlice(w.hidden, w.heads, w.ffn, w.layer_begin, w.layer_begin + w.layers,
                      B, w.seq, w.dtype, eps) as s:
        for i, p in enumerate(params):
            s.set_params(w.layer_begin + i, p)
        s.set_profiling(profiling)
        x = to_device(X, w.dtype)
        ln = torch.from_numpy(np.asarray(lens, np.int32)).cuda()
        dy = to_device(dY, w.dtype)
        if graph:
            y, dx = torch.empty_like(x), torch.empty_like(x)
            s.step_graph(x, ln, y, dy, dx)
            s.sync()
            for _ in range(steps):
                y.zero_()
                dx.zero_()
                s.launch_step_graph()
        else:
            for _ in range(steps):
                y = s.forward(x, ln)
                dx = s.backward(dy)
        s.sync()
        grads = [s.get_grads(w.layer_begin + i) for i in range(len(params))]
        return to_host(y), to_host(dx), grads


def compare_slice(w, Y, dX, grads, Yo, dXo, grads_o, rows=None):
    """Asserts every output tensor within the workload's tolerance; returns a report."""
    rep = {}
    sel = (slice(None),) if rows is None else (rows,)
    rep["Y"] = assert_close("Y", Y[sel], Yo, w.dtype)
    rep["dX"] = assert_close("dX", dX[sel], dXo, w.dtype)
    for i, (g, go) in enumerate(zip(grads, grads_o)):
        for k in ORC.PARAM_NAMES:
            rep[f"L{i}.{k}"] = assert_close(f"layer {i} grad {k}", g[k], go[k], w.dtype)
    return rep


def oracle_slice(w, X, lens, dY, params, eps=1e-12):
    return ORC.slice_step(np.asarray(X, np.float64), np.asarray(lens), np.asarray(dY, np.float64),
                          [{k: np.asarray(v, np.float64) for k, v in p.items()} for p in params],
                          w.heads, eps)


def oracle_slice_by_sequence(w, X, lens, dY, params, eps=1e-12):
    """The oracle's slice step on the whole batch, one sequence at a time.

    Each sequence's output and input gradient depend on that sequence alone
    (attention mixes only within a sequence; every other step acts row by
    row), and every weight gradient is a sum over the batch's rows, so the
    per-sequence weight gradients are added here in sequence order.  This
    keeps only one sequence's activation caches in host memory at a time."""
    B = X.shape[0]
    Y = np.empty(X.shape, np.float64)
    dX = np.empty(X.shape, np.float64)
    total = None
    for b in range(B):
        Yb, dXb, gb = oracle_slice(w, X[b:b + 1], lens[b:b + 1], dY[b:b + 1], params, eps)
        Y[b], dX[b] = Yb[0], dXb[0]
        if total is None:
            total = gb
        else:
            for acc, g in zip(total, gb):
                for k in acc:
                    acc[k] = acc[k] + g[k]
    return Y, dX, total
