"""A model split over devices by a partition index, run as a chain of slices.

Sky Computing trains a deep model by giving device ``i`` the layers
``pi[i] .. pi[i+1]-1`` (Sec. IV-D): the forward pass hands each device's
output to the next device and the backward pass runs in reverse order, every
device updating its own layers (Sec. III).  ``Pipeline`` builds that chain
out of ``EncoderSlice`` objects on one GPU and runs it for real, timing every
stage's forward and backward pass with CUDA events.

Heterogeneity is emulated as the paper's experiments do it (Sec. V-B): a
device with slow-down factor ``f`` takes ``f`` times its stage's time.

``step`` runs the stages one after another on one stream (one micro-batch),
timing each stage.  ``gpipe_makespan`` gives, from such stage times, the time
of one training step when D devices work in parallel on M micro-batches
(all forward passes, then all backward passes).  ``run_gpipe`` executes that
schedule: every stage has a CUDA stream of its own, a slice with one
activation stash per micro-batch, and events for the hand-offs; after every
forward or backward pass of a stage with slow-down ``f`` the stage's stream
is held for ``(f - 1)`` times the stage's calibrated time
(``sky_device_delay``), so the streams of faster stages go on while it waits.
The gradients of the micro-batches are summed in micro-batch order.
"""
from __future__ import annotations


def gpipe_makespan(fwd, bwd, micro_batches: int) -> float:
    """Time of one step of a D-stage pipeline on M micro-batches.

    ``fwd[i]`` / ``bwd[i]``: stage ``i``'s time per micro-batch.  Stage ``i``
    starts micro-batch ``m``'s forward when stage ``i-1`` has finished it and
    stage ``i`` has finished micro-batch ``m-1``; the backward passes start
    when every forward has finished and run from the last stage back, stage
    ``i`` starting micro-batch ``m``'s backward when stage ``i+1`` has
    finished it and stage ``i`` has finished micro-batch ``m-1``'s."""
    D, M = len(fwd), micro_batches
    if M < 1 or D < 1 or len(bwd) != D:
        raise ValueError("need D >= 1 stages with forward and backward times and M >= 1")
    f_end = [[0.0] * M for _ in range(D)]
    for i in range(D):
        for m in range(M):
            ready = max(f_end[i - 1][m] if i > 0 else 0.0, f_end[i][m - 1] if m > 0 else 0.0)
            f_end[i][m] = ready + fwd[i]
    start = f_end[D - 1][M - 1]
    b_end = [[0.0] * M for _ in range(D)]
    for i in reversed(range(D)):
        for m in range(M):
            ready = max(b_end[i + 1][m] if i + 1 < D else start,
                        b_end[i][m - 1] if m > 0 else start)
            b_end[i][m] = ready + bwd[i]
    return b_end[0][M - 1]


class Pipeline:
    """Layers ``[pi[0], pi[-1])`` of a post-LN BERT encoder split into D slices.

    ``params[l]`` holds the 12 tensors of global layer ``l``.  Hand-offs
    between slices are fp32 (``io_fp32``), so the chain reproduces one slice
    over all the layers bit for bit."""

    def __init__(self, width, heads, ffn, pi, params, max_batch, seq, dtype="bf16",
                 micro_batches: int = 1):
        from .slice import EncoderSlice
        self.pi = list(pi)
        self.stages = []
        self.M = micro_batches
        for i in range(len(pi) - 1):
            s = EncoderSlice(width, heads, ffn, pi[i], pi[i + 1], max_batch, seq, dtype,
                             io_fp32=dtype == "bf16", stash_slots=micro_batches)
            for l in range(pi[i], pi[i + 1]):
                s.set_params(l, params[l])
            self.stages.append(s)

    def close(self):
        for s in self.stages:
            s.close()
        self.stages = []

    def __enter__(self):
        return self

    def __exit__(self, *a):
        self.close()

    def step(self, x, lens, dy):
        """Forward through every stage, then backward in reverse.

        ``x`` and ``dy`` are fp32 device tensors ``[B, S, H]`` for a bf16
        chain (the slice dtype for fp32).  Returns ``(y, dx, fwd_ms, bwd_ms)``
        with per-stage CUDA-event times."""
        import torch
        stream = torch.cuda.current_stream()
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(2 * len(self.stages))]
        h = x
        for i, s in enumerate(self.stages):
            ev[i][0].record(stream)
            h = s.forward(h, lens, stream=stream)
            ev[i][1].record(stream)
        y = h
        g = dy
        for i in reversed(range(len(self.stages))):
            k = len(self.stages) + i
            ev[k][0].record(stream)
            g = self.stages[i].backward(g, stream=stream)
            ev[k][1].record(stream)
        torch.cuda.synchronize()
        D = len(self.stages)
        fwd = [ev[i][0].elapsed_time(ev[i][1]) for i in range(D)]
        bwd = [ev[D + i][0].elapsed_time(ev[D + i][1]) for i in range(D)]
        return y, g, fwd, bwd

    def grads(self, layer: int) -> dict:
        i = max(k for k in range(len(self.pi) - 1) if self.pi[k] <= layer)
        return self.stages[i].get_grads(layer)

    def run_gpipe(self, xs, lens, dys, slow=None, fwd_ms=None, bwd_ms=None):
        """Executes one GPipe step over ``M = len(xs)`` micro-batches.

        ``xs[m]``, ``dys[m]``: device tensors ``[B, S, H]`` (fp32 for a bf16
        chain), ``lens[m]`` device int32 ``[B]``.  ``slow[i]`` is stage i's
        slow-down factor (default 1) and ``fwd_ms[i]`` / ``bwd_ms[i]`` its
        calibrated per-micro-batch times, from which the emulation delays are
        formed.  Stage i runs forward(m) after stage i-1 has, for m = 0..M-1,
        then backward(m) after stage i+1 has, for m = 0..M-1, with
        micro-batch m's activations in stash slot m and gradients summed in
        micro-batch order (the first overwrites).  Returns ``(ys, dxs,
        makespan_ms)``: per micro-batch output and input gradient, and the
        wall time of the whole step between CUDA events."""
        import torch
        from . import _lib as L
        D, M = len(self.stages), len(xs)
        if M > self.M or len(lens) != M or len(dys) != M:
            raise ValueError(f"need M <= {self.M} micro-batches with lengths and gradients")
        slow = list(slow) if slow is not None else [1.0] * D
        if (any(f > 1.0 for f in slow)) and (fwd_ms is None or bwd_ms is None):
            raise ValueError("slow-down emulation needs the calibrated stage times")
        cur = torch.cuda.current_stream()
        streams = [torch.cuda.Stream() for _ in range(D)]
        ev = lambda: torch.cuda.Event()
        f_done = [[ev() for _ in range(M)] for _ in range(D)]
        b_done = [[ev() for _ in range(M)] for _ in range(D)]
        t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

        def delay(i, ms, st):
            ns = int(round((slow[i] - 1.0) * ms * 1e6))
            if ns > 0:
                L.call("sky_device_delay", ns, int(st.cuda_stream))

        h = [[None] * M for _ in range(D)]
        g = [[None] * M for _ in range(D)]
        t0.record(cur)
        for st in streams:
            st.wait_stream(cur)
        for m in range(M):
            for i, s in enumerate(self.stages):
                st = streams[i]
                with torch.cuda.stream(st):
                    if i > 0:
                        st.wait_event(f_done[i - 1][m])
                    inp = xs[m] if i == 0 else h[i - 1][m]
                    h[i][m] = s.forward(inp, lens[m], stream=st, slot=m)
                    if slow[i] > 1.0:
                        delay(i, fwd_ms[i], st)
                    f_done[i][m].record(st)
        for m in range(M):
            for i in reversed(range(D)):
                st = streams[i]
                with torch.cuda.stream(st):
                    if i + 1 < D:
                        st.wait_event(b_done[i + 1][m])
                    grad = dys[m] if i + 1 == D else g[i + 1][m]
                    g[i][m] = self.stages[i].backward(grad, stream=st, slot=m, accumulate=m > 0)
                    if slow[i] > 1.0:
                        delay(i, bwd_ms[i], st)
                    b_done[i][m].record(st)
        for st in streams:
            cur.wait_stream(st)
        t1.record(cur)
        t1.synchronize()
        for s in self.stages:
            s.sync()
        return [h[D - 1][m] for m in range(M)], [g[0][m] for m in range(M)], t0.elapsed_time(t1)
