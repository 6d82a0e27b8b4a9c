"""Slice-level parity: the whole forward + backward of an encoder slice on the
GPU (through sky_slice.h) against the float64 oracle on the same seeded
inputs, every output tensor (Y, dX and the 12 gradients of every layer).

Every case compares the whole batch.  At the full-size workloads the oracle
runs one sequence at a time (a sequence's forward and input gradient depend
on it alone, and weight gradients are sums over sequences), while the GPU runs
the whole batch in the benchmark's launch configuration.
"""
import numpy as np
import pytest

from paper_2202_11836_gb300 import synth
from parity_util import (compare_slice, oracle_slice, oracle_slice_by_sequence, run_gpu_slice,
                         to_device, to_host)

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")


def full_case(w, affine="random"):
    params = synth.slice_params(w, affine=affine)
    X, lens, dY = synth.activations(w), synth.lengths(w), synth.upstream_grad(w)
    Y, dX, grads = run_gpu_slice(w, X, lens, dY, params, None)
    Yo, dXo, go = oracle_slice(w, X, lens, dY, params)
    return compare_slice(w, Y, dX, grads, Yo, dXo, go)


def test_tiny_fp32_slice():
    """2-layer fp32 slice (H=128, A=2, F=512, S=32, B=4): maxrel <= 1e-4."""
    full_case(synth.WORKLOADS["tiny-fp32"])
    full_case(synth.WORKLOADS["tiny-fp32"], affine="bert")


@pytest.mark.parametrize("w", [
    synth.custom("bf16-ragged", layers=2, hidden=256, heads=4, ffn=1024, seq=96, batch=3,
                 len_lo=1, len_hi=96, dy_std=1e-2),
    synth.custom("bf16-odd-tail", layers=1, hidden=128, heads=2, ffn=520, seq=77, batch=5,
                 len_lo=1, len_hi=77, dy_std=1e-2),
    synth.custom("bf16-s1", layers=1, hidden=128, heads=2, ffn=256, seq=1, batch=8,
                 len_lo=1, len_hi=1, dy_std=1e-2),
], ids=lambda w: w.name)
def test_bf16_small_slices(w):
    full_case(w)


def test_base_width_slice_full():
    """BERT-base width, 4 layers, S=128, B=32: every sequence checked."""
    full_case(synth.WORKLOADS["base-s128"], affine="bert")


def full_batch_case(w):
    """The whole batch on both sides, with the workload's upstream gradient on
    every sequence: the GPU runs the step as the benchmark times it (captured
    once as a CUDA graph and replayed into zeroed outputs); the oracle runs
    sequence by sequence.  Every row of Y and dX and every gradient of every
    layer is compared."""
    params = synth.slice_params(w, affine="bert")
    X, lens, dY = synth.activations(w), synth.lengths(w), synth.upstream_grad(w)
    Y, dX, grads = run_gpu_slice(w, X, lens, dY, params, None, graph=True)
    Yo, dXo, go = oracle_slice_by_sequence(w, X, lens, dY, params)
    rep = compare_slice(w, Y, dX, grads, Yo, dXo, go)
    worst = max(rep.items(), key=lambda kv: kv[1][1])
    print(f"\n{w.name}: worst l2rel {worst[1][1]:.2e} ({worst[0]}), "
          f"worst maxrel {max(v[0] for v in rep.values()):.2e}")
    return rep


def test_large_width_slice_full_batch():
    """BERT-large width, 8 layers, S=512, B=16 (the benchmark workload): all
    16 sequences, every output tensor."""
    full_batch_case(synth.WORKLOADS["large-s512"])


def test_long_sequence_slice_full_batch():
    """S=2048, B=4, 4 layers (two full-length sequences, two ragged): all 4
    sequences, every output tensor."""
    full_batch_case(synth.WORKLOADS["large-s2048"])


def test_padding_gradient_isolation_at_full_size():
    """Full-size batch with the upstream gradient zeroed on all but two
    sequences: those two match the oracle run on them alone, and the other
    sequences receive an input gradient of exactly zero."""
    w = synth.WORKLOADS["large-s512"]
    lens = synth.lengths(w)
    sample = (int(np.argmin(lens)), int(np.argmax(lens)))
    params = synth.slice_params(w, affine="bert")
    X, dY = synth.activations(w), synth.upstream_grad(w)
    mask = np.zeros(w.batch, bool)
    mask[list(sample)] = True
    dY = dY * mask[:, None, None]
    Y, dX, grads = run_gpu_slice(w, X, lens, dY, params, None, graph=True)
    idx = np.array(sample)
    Yo, dXo, go = oracle_slice(w, X[idx], lens[idx], dY[idx], params)
    compare_slice(w, Y, dX, grads, Yo, dXo, go, rows=idx)
    rest = np.where(~mask)[0]
    assert np.all(dX[rest] == 0.0)


def _slice_run(w, lb, le, X, lens, dY, params, io_fp32=False):
    from paper_2202_11836_gb300.slice import EncoderSlice
    dt = "fp32" if io_fp32 else w.dtype
    with EncoderSlice(w.hidden, w.heads, w.ffn, lb, le, w.batch, w.seq, w.dtype,
                      io_fp32=io_fp32) as s:
        for l in range(lb, le):
            s.set_params(l, params[l])
        x = X if torch.is_tensor(X) else to_device(X, dt)
        ln = torch.from_numpy(lens).cuda()
        y = s.forward(x, ln)
        dx = s.backward(dY if torch.is_tensor(dY) else to_device(dY, dt))
        s.sync()
        return y, dx, [s.get_grads(l) for l in range(lb, le)]


def test_uneven_slices_compose_bitwise():
    """With fp32 boundary tensors, slices [0,1) then [1,4) of the 160-layer
    base-width model reproduce slice [0,4) bit for bit (forward, input
    gradient and every weight gradient); with bf16 boundaries they agree
    within the bf16 tolerance (one rounding of the hand-off tensor)."""
    from parity_util import assert_close
    w = synth.WORKLOADS["base-s128-b16"]
    params = {l: synth.layer_params(l, w.hidden, w.ffn, "bf16", affine="random") for l in range(4)}
    X, lens, dY = synth.activations(w), synth.lengths(w), synth.upstream_grad(w)
    for io32 in (True, False):
        y_full, dx_full, g_full = _slice_run(w, 0, 4, X, lens, dY, params, io32)
        y1, _, _ = _slice_run(w, 0, 1, X, lens, dY, params, io32)
        y2, dmid, g2 = _slice_run(w, 1, 4, y1, lens, dY, params, io32)
        _, dx1, g1 = _slice_run(w, 0, 1, X, lens, dmid, params, io32)
        if io32:
            assert y_full.dtype == torch.float32
            assert torch.equal(y2, y_full)
            assert torch.equal(dx1, dx_full)
            for a, b in zip(g1 + g2, g_full):
                for k in a:
                    assert np.array_equal(a[k], b[k]), k
        else:
            assert_close("y", to_host(y2), to_host(y_full), "bf16")
            assert_close("dx", to_host(dx1), to_host(dx_full), "bf16")
            for a, b in zip(g1 + g2, g_full):
                for k in a:
                    assert_close(k, a[k], b[k], "bf16")


def test_uneven_slice_parity():
    """The 7-layer slice [4, 11) of the 160-layer base-width model vs the oracle."""
    w0 = synth.WORKLOADS["base-s128-b16"]
    import dataclasses
    w = dataclasses.replace(w0, layers=7, layer_begin=4)
    full_case(w, affine="bert")


def test_deterministic_and_status():
    from paper_2202_11836_gb300 import _lib as L
    from paper_2202_11836_gb300.slice import EncoderSlice
    w = synth.custom("det", layers=2, hidden=256, heads=4, ffn=512, seq=64, batch=4, len_lo=1,
                     len_hi=64)
    params = synth.slice_params(w, affine="random")
    X, lens, dY = synth.activations(w), synth.lengths(w), synth.upstream_grad(w)
    a = run_gpu_slice(w, X, lens, dY, params, None)
    b = run_gpu_slice(w, X, lens, dY, params, None)
    assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1])
    with EncoderSlice(256, 4, 512, 0, 2, 4, 64) as s:
        x = to_device(X, "bf16")
        dy = to_device(dY, "bf16")
        with pytest.raises(L.SkyError) as e:
            s.backward(dy)
        assert e.value.status == L.SKY_ERR_STATE
        bad = torch.tensor([0, 5, 64, 65], dtype=torch.int32, device="cuda")
        s.forward(x, bad)
        with pytest.raises(L.SkyError) as e:
            s.sync()
        assert e.value.status == L.SKY_ERR_INVALID_ARG
        s.sync()  # status word was cleared
        with pytest.raises(L.SkyError) as e:
            s.forward(torch.zeros((5, 64, 256), dtype=torch.bfloat16, device="cuda"), bad)
        assert e.value.status == L.SKY_ERR_INVALID_ARG


def test_fp32_input_read_in_place_or_copied():
    """A bf16 slice with fp32 boundary tensors reads an aligned x in place as
    the first layer's residual and copies a misaligned one first.  Both give
    the same bits (forward, input gradient, every weight gradient), and x is
    left unchanged."""
    w = synth.custom("x-align", layers=2, hidden=256, heads=4, ffn=512, seq=64, batch=4,
                     len_lo=1, len_hi=64, dy_std=1e-2)
    params = synth.slice_params(w, affine="random")
    X, lens, dY = synth.activations(w), synth.lengths(w), synth.upstream_grad(w)
    xa = to_device(X, "fp32")
    n = xa.numel()
    buf = torch.empty(n + 1, dtype=torch.float32, device="cuda")
    xm = buf[1:].view(xa.shape)  # 4 bytes past a 16-byte boundary
    xm.copy_(xa)
    assert xm.data_ptr() % 16 == 4
    ya, dxa, ga = _slice_run(w, 0, 2, xa, lens, dY, params, io_fp32=True)
    ym, dxm, gm = _slice_run(w, 0, 2, xm, lens, dY, params, io_fp32=True)
    assert torch.equal(ya, ym) and torch.equal(dxa, dxm)
    for a, b in zip(ga, gm):
        for k in a:
            assert np.array_equal(a[k], b[k]), k
    assert torch.equal(xa.cpu(), torch.from_numpy(np.asarray(X, np.float32)))
    assert torch.equal(xm, xa)


def test_side_stream_backward_matches_in_line():
    """The bf16 backward runs its weight-gradient GEMMs on a second stream that
    overlaps the data-gradient chain and reuses shared gradient buffers across
    layers.  Two back-to-back steps with that overlap must reproduce, bit for
    bit, the backward with every kernel in line on the caller's stream."""
    w = synth.custom("side", layers=3, hidden=1024, heads=16, ffn=4096, seq=256, batch=8,
                     len_lo=128, len_hi=256)
    params = synth.slice_params(w, affine="random")
    X, lens, dY = synth.activations(w), synth.lengths(w), synth.upstream_grad(w)
    a = run_gpu_slice(w, X, lens, dY, params, None, steps=2)
    b = run_gpu_slice(w, X, lens, dY, params, None, steps=1, profiling=True)
    assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1])
    for ga, gb in zip(a[2], b[2]):
        for k in ga:
            assert np.array_equal(ga[k], gb[k]), k


def test_layer_cost_and_linearity():
    """Per-layer cost records and slice time linear in the number of layers."""
    import time
    from paper_2202_11836_gb300.slice import EncoderSlice
    w = synth.WORKLOADS["base-s128-b16"]
    times = []
    for (lb, le) in synth.UNEVEN_SLICES:
        with EncoderSlice(w.hidden, w.heads, w.ffn, lb, le, w.batch, w.seq) as s:
            for l in range(lb, le):
                s.set_params(l, synth.layer_params(l, w.hidden, w.ffn, "bf16"))
            rec = s.layer_cost(w.batch, w.seq, iters=3, lens=synth.lengths(w))
            assert len(rec) == le - lb
            for r in rec:
                assert r["fwd_ms"] > 0 and r["bwd_ms"] > 0
                assert r["param_bytes"] == 2 * (4 * 768 * 768 + 2 * 768 * 3072 + 9 * 768 + 3072)
            times.append(sum(r["fwd_ms"] + r["bwd_ms"] for r in rec))
    n = np.array([le - lb for lb, le in synth.UNEVEN_SLICES], float)
    t = np.array(times)
    beta, alpha = np.polyfit(n, t, 1)
    pred = alpha + beta * n
    r2 = 1 - ((t - pred) ** 2).sum() / ((t - t.mean()) ** 2).sum()
    assert r2 >= 0.99, (times, r2)


def test_layer_cost_counts_the_mask_and_waits_for_queued_work():
    """sky_slice_layer_cost measures the workload's own lengths (its attention
    FLOPs count the valid keys) and rejects a length outside [1, S].  Called
    right after a step that is still queued on the caller's stream, it first
    waits for that step: the step's y and dx equal those of the same step run
    alone."""
    from paper_2202_11836_gb300 import _lib as L
    from paper_2202_11836_gb300.slice import EncoderSlice
    w = synth.custom("cost", layers=2, hidden=1024, heads=16, ffn=4096, seq=512, batch=8,
                     len_lo=100, len_hi=512)
    params = synth.slice_params(w, affine="random")
    X, lens, dY = synth.activations(w), synth.lengths(w), synth.upstream_grad(w)
    T, H, F, S = w.batch * w.seq, w.hidden, w.ffn, w.seq
    with EncoderSlice(H, w.heads, F, 0, w.layers, w.batch, S) as s:
        for i, p in enumerate(params):
            s.set_params(i, p)
        x, dy = to_device(X, "bf16"), to_device(dY, "bf16")
        ln = torch.from_numpy(lens).cuda()
        y_ref = s.forward(x, ln).clone()
        dx_ref = s.backward(dy).clone()
        s.sync()
        y, dx = torch.empty_like(x), torch.empty_like(x)
        s.forward(x, ln, y)
        s.backward(dy, dx)
        rec = s.layer_cost(w.batch, S, iters=2, lens=lens)  # no sync before it
        torch.cuda.synchronize()
        assert torch.equal(y, y_ref) and torch.equal(dx, dx_ref)
        gemm = 2.0 * T * (4 * H * H + 2 * H * F)
        for r in rec:
            assert r["fwd_flops"] == pytest.approx(gemm + 4.0 * H * S * lens.sum(), rel=1e-12)
            assert r["bwd_flops"] == pytest.approx(2 * r["fwd_flops"], rel=1e-12)
        full = s.layer_cost(w.batch, S, iters=2)
        assert full[0]["fwd_flops"] == pytest.approx(gemm + 4.0 * H * S * S * w.batch, rel=1e-12)
        bad = lens.copy()
        bad[1] = S + 1
        with pytest.raises(L.SkyError) as e:
            s.layer_cost(w.batch, S, iters=1, lens=bad)
        assert e.value.status == L.SKY_ERR_INVALID_ARG


def test_layer_cost_feeds_allocator():
    """The per-layer records of sky_slice_layer_cost are the model benchmark
    of Sec. IV-B: their time and bytes form the allocator's layer table, and
    a slow device gets fewer layers than a fast one."""
    from paper_2202_11836_gb300 import allocator
    from paper_2202_11836_gb300.slice import EncoderSlice
    w = synth.WORKLOADS["base-s128-b16"]
    lb, le = 0, 6
    with EncoderSlice(w.hidden, w.heads, w.ffn, lb, le, w.batch, w.seq) as s:
        for l in range(lb, le):
            s.set_params(l, synth.layer_params(l, w.hidden, w.ffn, "bf16"))
        rec = s.layer_cost(w.batch, w.seq, iters=3, lens=synth.lengths(w))
    lf, lm = allocator.layer_table(rec)
    assert all(f > 0 for f in lf) and all(m > 0 for m in lm)
    t = [r["fwd_ms"] + r["bwd_ms"] for r in rec]
    # three devices, the middle one three times slower; memory for 4 layers each
    P = allocator.Problem([1.0, 3.0, 1.0], [4 * max(lm)] * 3, [0.0] * 3, t, lm)
    pi = P.heuristic()
    counts = [pi[i + 1] - pi[i] for i in range(3)]
    assert pi[0] == 0 and pi[-1] == le - lb and min(counts) >= 1
    assert counts[1] <= min(counts[0], counts[2])
    assert P.makespan(pi) <= P.makespan(allocator.even(le - lb, 3))


@pytest.mark.parametrize("wname", ["base-s128", "tiny-fp32"])
def test_step_graph_replays_direct_step_bitwise(wname):
    """The captured training step (sky_slice_step_graph_create / _launch)
    reproduces a direct forward + backward bit for bit (output, input
    gradient, every layer's gradients) on inputs refilled in place after the
    capture, over two replays, and counts the same kernel launches."""
    from paper_2202_11836_gb300 import _lib as L
    from paper_2202_11836_gb300.slice import EncoderSlice
    w = synth.WORKLOADS[wname]
    params = synth.slice_params(w, affine="random")
    X, lens, dY = synth.activations(w), synth.lengths(w), synth.upstream_grad(w)
    X2 = synth.activations(w, seed=synth.SEED + 1)
    dY2 = synth.upstream_grad(w, seed=synth.SEED + 1)
    lens2 = synth.lengths(w, seed=synth.SEED + 1)
    lib = L.lib()
    with EncoderSlice(w.hidden, w.heads, w.ffn, 0, w.layers, w.batch, w.seq, w.dtype) as s:
        for i, p in enumerate(params):
            s.set_params(i, p)
        # direct step on the second inputs: the reference
        n0 = lib.sky_launch_count()
        y_ref = s.forward(to_device(X2, w.dtype), torch.from_numpy(lens2).cuda())
        dx_ref = s.backward(to_device(dY2, w.dtype))
        s.sync()
        per_step = lib.sky_launch_count() - n0
        g_ref = [s.get_grads(i) for i in range(w.layers)]
        # capture on the first inputs, then refill them in place
        x = to_device(X, w.dtype)
        ln = torch.from_numpy(lens).cuda()
        dy = to_device(dY, w.dtype)
        y, dx = torch.empty_like(x), torch.empty_like(x)
        s.step_graph(x, ln, y, dy, dx)
        s.sync()
        x.copy_(to_device(X2, w.dtype))
        dy.copy_(to_device(dY2, w.dtype))
        ln.copy_(torch.from_numpy(lens2))
        for _ in range(2):
            y.zero_()
            dx.zero_()
            n1 = lib.sky_launch_count()
            s.launch_step_graph()
            s.sync()
            assert lib.sky_launch_count() - n1 == per_step
            assert torch.equal(y, y_ref) and torch.equal(dx, dx_ref)
            for i in range(w.layers):
                g = s.get_grads(i)
                for k in g:
                    assert np.array_equal(g[k], g_ref[i][k]), (i, k)
        # with per-kernel timing on, the captured step times every kernel at
        # each replay and still gives the same bits
        s.set_profiling(True)
        s.step_graph(x, ln, y, dy, dx)
        for _ in range(2):
            y.zero_()
            s.launch_step_graph()
        s.sync()
        assert torch.equal(y, y_ref)
        stats = s.kernel_stats()
        n_rec = sum(v["launches"] for v in stats.values())
        assert n_rec > 0 and n_rec % 2 == 0
        assert all(v["total_ms"] > 0 for v in stats.values())
        s.set_profiling(False)
