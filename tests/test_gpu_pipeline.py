"""A 12-layer model split over four emulated devices (Sec. III, IV-D, V-A).

The chain of slices built from a partition index must reproduce one slice
over all the layers bit for bit (fp32 hand-offs).  With the paper's
slow-down emulation (device i takes f_i times the measured stage time), the
heuristic allocation computed from measured per-layer costs gives a shorter
pipelined step than the even split -- the shape of the paper's comparison,
on synthetic data and one GPU."""
import numpy as np
import pytest

from paper_2202_11836_gb300 import synth

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")


def test_pipeline_composes_and_heuristic_beats_even():
    from paper_2202_11836_gb300 import allocator
    from paper_2202_11836_gb300.pipeline import Pipeline, gpipe_makespan
    from paper_2202_11836_gb300.slice import EncoderSlice
    w = synth.custom("pipe", layers=12, hidden=768, heads=12, ffn=3072, seq=128, batch=8,
                     len_lo=64, len_hi=128)
    L = w.layers
    params = synth.slice_params(w, affine="random")
    X, lens, dY = synth.activations(w), synth.lengths(w), synth.upstream_grad(w)
    x = torch.from_numpy(X.astype(np.float32)).cuda()
    dy = torch.from_numpy(dY.astype(np.float32)).cuda()
    ln = torch.from_numpy(np.asarray(lens, np.int32)).cuda()
    B = X.shape[0]

    # the whole model as one slice: reference outputs and per-layer costs
    with EncoderSlice(w.hidden, w.heads, w.ffn, 0, L, B, w.seq, io_fp32=True) as s:
        for l in range(L):
            s.set_params(l, params[l])
        y_ref = s.forward(x, ln).cpu().numpy()
        dx_ref = s.backward(dy).cpu().numpy()
        g_ref = [s.get_grads(l) for l in range(L)]
        costs = s.layer_cost(B, w.seq, iters=3, lens=lens)

    slow = [1.0, 2.0, 4.0, 7.0]
    t_layer = [r["fwd_ms"] + r["bwd_ms"] for r in costs]
    _, lm = allocator.layer_table(costs)
    P = allocator.Problem(slow, [L * max(lm)] * 4, [0.0] * 4, t_layer, lm)
    plans = {"even": allocator.even(L, 4), "heuristic": P.heuristic()}
    makespan = {}
    for name, pi in plans.items():
        with Pipeline(w.hidden, w.heads, w.ffn, pi, params, B, w.seq) as pipe:
            pipe.step(x, ln, dy)  # warm-up
            y, dx, fwd, bwd = pipe.step(x, ln, dy)
            assert np.array_equal(y.cpu().numpy(), y_ref), name
            assert np.array_equal(dx.cpu().numpy(), dx_ref), name
            for l in range(L):
                g = pipe.grads(l)
                for k in g:
                    assert np.array_equal(g[k], g_ref[l][k]), (name, l, k)
        makespan[name] = gpipe_makespan([f * a for f, a in zip(slow, fwd)],
                                        [f * b for f, b in zip(slow, bwd)], 8)
    print(f"\nplans {plans}; emulated step (8 micro-batches): even {makespan['even']:.2f} ms, "
          f"heuristic {makespan['heuristic']:.2f} ms")
    assert makespan["heuristic"] < makespan["even"]
