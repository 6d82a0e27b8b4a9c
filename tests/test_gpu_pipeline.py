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


def _micro_batches(w, M, B):
    """M seeded micro-batches of B sequences each (fp32 hand-off tensors)."""
    xs, lens, dys = [], [], []
    for m in range(M):
        seed = synth.SEED + 100 + m
        xs.append(torch.from_numpy(synth.activations(w, seed=seed, batch=B).astype(np.float32)).cuda())
        lens.append(torch.from_numpy(synth.lengths(w, seed=seed, batch=B)).cuda())
        dys.append(torch.from_numpy(synth.upstream_grad(w, seed=seed, batch=B).astype(np.float32)).cuda())
    return xs, lens, dys


def test_stash_slots_accumulate_bitwise():
    """Three forwards into stash slots 0, 1, 2, then their backwards in the
    order 1, 0, 2 (the first overwriting the gradients, the others adding):
    every output and input gradient equals that micro-batch's own step, and
    the gradients equal the ones obtained by running the three steps one
    after another with the same accumulation order (bitwise).  A backward
    into a slot without a forward is a STATE error."""
    from paper_2202_11836_gb300 import _lib as L
    from paper_2202_11836_gb300.slice import EncoderSlice
    w = synth.custom("slots", layers=2, hidden=768, heads=12, ffn=3072, seq=128, batch=4,
                     len_lo=16, len_hi=128)
    params = synth.slice_params(w, affine="random")
    xs, lens, dys = _micro_batches(w, 3, 4)
    order = (1, 0, 2)
    with EncoderSlice(w.hidden, w.heads, w.ffn, 0, 2, 4, w.seq, io_fp32=True, stash_slots=3) as s:
        for l in range(2):
            s.set_params(l, params[l])
        # reference: one step at a time, same accumulation order
        ref_y, ref_dx = {}, {}
        for k, m in enumerate(order):
            ref_y[m] = s.forward(xs[m], lens[m], slot=0).clone()
            ref_dx[m] = s.backward(dys[m], slot=0, accumulate=k > 0).clone()
        s.sync()
        ref_g = [s.get_grads(l) for l in range(2)]
        # all forwards first, then the backwards
        ys = {m: s.forward(xs[m], lens[m], slot=m) for m in range(3)}
        dxs = {}
        for k, m in enumerate(order):
            dxs[m] = s.backward(dys[m], slot=m, accumulate=k > 0)
        s.sync()
        for m in range(3):
            assert torch.equal(ys[m], ref_y[m]) and torch.equal(dxs[m], ref_dx[m]), m
        for l in range(2):
            g = s.get_grads(l)
            for k in g:
                assert np.array_equal(g[k], ref_g[l][k]), (l, k)
    with EncoderSlice(w.hidden, w.heads, w.ffn, 0, 1, 4, w.seq, io_fp32=True, stash_slots=2) as s:
        with pytest.raises(L.SkyError) as e:
            s.backward(dys[0], slot=1)
        assert e.value.status == L.SKY_ERR_STATE
    with EncoderSlice(w.hidden, w.heads, w.ffn, 0, 1, 4, w.seq, io_fp32=True) as s:
        s.forward(xs[0], lens[0])
        with pytest.raises(L.SkyError) as e:
            s.backward(dys[0], accumulate=True)
        assert e.value.status == L.SKY_ERR_UNSUPPORTED


def test_gpipe_schedule_executed():
    """The GPipe schedule of 4 micro-batches over 4 emulated devices
    (slow-down 1, 2, 4, 7), executed with one stream per stage: every
    micro-batch's output and input gradient, and the summed gradients, equal
    the unsplit 12-layer slice run one micro-batch at a time (bitwise); the
    executed step time is close to the GPipe makespan computed from the
    calibrated stage times; the heuristic partition's executed step is
    shorter than the even split's."""
    from paper_2202_11836_gb300 import allocator
    from paper_2202_11836_gb300.pipeline import Pipeline, gpipe_makespan
    from paper_2202_11836_gb300.slice import EncoderSlice
    w = synth.custom("gpipe", layers=12, hidden=768, heads=12, ffn=3072, seq=128, batch=8,
                     len_lo=64, len_hi=128)
    L_, M, B = w.layers, 4, 8
    params = synth.slice_params(w, affine="random")
    xs, lens, dys = _micro_batches(w, M, B)
    slow = [1.0, 2.0, 4.0, 7.0]
    with EncoderSlice(w.hidden, w.heads, w.ffn, 0, L_, B, w.seq, io_fp32=True) as s:
        for l in range(L_):
            s.set_params(l, params[l])
        costs = s.layer_cost(B, w.seq, iters=3, lens=synth.lengths(w, batch=B))
    with EncoderSlice(w.hidden, w.heads, w.ffn, 0, L_, B, w.seq, io_fp32=True, stash_slots=2) as s:
        for l in range(L_):
            s.set_params(l, params[l])
        ref_y, ref_dx = [], []
        for m in range(M):
            ref_y.append(s.forward(xs[m], lens[m]).clone())
            ref_dx.append(s.backward(dys[m], accumulate=m > 0).clone())
        s.sync()
        ref_g = [s.get_grads(l) for l in range(L_)]
    t_layer = [r["fwd_ms"] + r["bwd_ms"] for r in costs]
    _, lm = allocator.layer_table(costs)
    P = allocator.Problem(slow, [L_ * max(lm)] * 4, [0.0] * 4, t_layer, lm)
    plans = {"even": allocator.even(L_, 4), "heuristic": P.heuristic()}
    executed, predicted = {}, {}
    for name, pi in plans.items():
        with Pipeline(w.hidden, w.heads, w.ffn, pi, params, B, w.seq, micro_batches=M) as pipe:
            # calibration: each stage alone, one micro-batch
            pipe.step(xs[0], lens[0], dys[0])
            _, _, fwd, bwd = pipe.step(xs[0], lens[0], dys[0])
            pipe.run_gpipe(xs, lens, dys, slow, fwd, bwd)  # warm-up
            ys, dxs, ms = pipe.run_gpipe(xs, lens, dys, slow, fwd, bwd)
            for m in range(M):
                assert torch.equal(ys[m], ref_y[m]), (name, m)
                assert torch.equal(dxs[m], ref_dx[m]), (name, m)
            for l in range(L_):
                g = pipe.grads(l)
                for k in g:
                    assert np.array_equal(g[k], ref_g[l][k]), (name, l, k)
        executed[name] = ms
        predicted[name] = gpipe_makespan([f * a for f, a in zip(slow, fwd)],
                                         [f * b for f, b in zip(slow, bwd)], M)
    print(f"\nplans {plans}; executed {executed}; GPipe makespan {predicted}")
    for name in plans:
        # stages that compute at the same time share the one GPU, so the executed
        # step is somewhat longer than the model of D separate devices
        assert 0.85 * predicted[name] <= executed[name] <= 1.4 * predicted[name], name
    assert executed["heuristic"] < executed["even"]
