"""A model split over devices by a partition index, run as a chain of slices.

Sky Computing trains a deep model by giving device ``i`` the layers
``pi[i] .. pi[i+1]-1`` (Sec. IV-D): the forward pass hands each device's
output to the next device and the backward pass runs in reverse order, every
device updating its own layers (Sec. III).  ``Pipeline`` builds that chain
out of ``EncoderSlice`` objects on one GPU and runs it for real, timing every
stage's forward and backward pass with CUDA events.

One GPU cannot run the stages at the same time, and it is one device, not a
set of heterogeneous ones.  Heterogeneity is emulated as the paper's
experiments do it (Sec. V-A): a device with slow-down factor ``f`` takes ``f``
times the measured time of its stage.  ``gpipe_makespan`` then gives the time
of one training step when the D devices work in parallel on M micro-batches
(all forward passes, then all backward passes), from those stage times.
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

    def __init__(self, width, heads, ffn, pi, params, max_batch, seq, dtype="bf16"):
        from .slice import EncoderSlice
        self.pi = list(pi)
        self.stages = []
        for i in range(len(pi) - 1):
            s = EncoderSlice(width, heads, ffn, pi[i], pi[i + 1], max_batch, seq, dtype,
                             io_fp32=dtype == "bf16")
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
