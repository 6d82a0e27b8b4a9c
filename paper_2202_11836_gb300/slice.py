"""Python view of one encoder slice: a handle on the C ABI of sky_slice.h.

PyTorch supplies device memory and the CUDA stream; every computation runs in
libsky_slice.so.  A slice owns the layers [layer_begin, layer_end) of a deep
post-LN BERT encoder (the contiguous layer range a device is assigned,
Sec. IV-D of the paper) and runs their forward and backward pass.
"""
from __future__ import annotations

import ctypes as C

import numpy as np

from . import _lib as L
from .synth import PARAM_NAMES, from_bf16_bits, to_bf16_bits


def _stream_ptr(stream) -> int:
    import torch
    s = stream if stream is not None else torch.cuda.current_stream()
    return int(s.cuda_stream)


def _ptr(t) -> int:
    return int(t.data_ptr())


class EncoderSlice:
    """Layers [layer_begin, layer_end) with hidden width H, A heads and FFN width F."""

    def __init__(self, width: int, heads: int, ffn: int, layer_begin: int, layer_end: int,
                 max_batch: int, max_seq: int, dtype: str = "bf16", ln_eps: float = 1e-12,
                 io_fp32: bool = False, stash_slots: int = 1):
        self.H, self.A, self.F = width, heads, ffn
        self.layer_begin, self.layer_end = layer_begin, layer_end
        self.dtype = dtype
        self.io_fp32 = io_fp32
        cfg = L.SkySliceConfig(width, heads, ffn, layer_begin, layer_end, max_batch, max_seq,
                               L.SKY_DTYPE_BF16 if dtype == "bf16" else L.SKY_DTYPE_FP32,
                               ln_eps, 1 if io_fp32 else 0, stash_slots)
        h = C.c_void_p()
        L.call("sky_slice_create", C.byref(cfg), C.byref(h))
        self.h = h
        self._fwd_keep = {}

    # ----------------------------------------------------------- parameters
    def shapes(self):
        H, F = self.H, self.F
        return {"Wqkv": (3 * H, H), "bqkv": (3 * H,), "Wo": (H, H), "bo": (H,),
                "gamma1": (H,), "beta1": (H,), "W1": (F, H), "b1": (F,), "W2": (H, F),
                "b2": (H,), "gamma2": (H,), "beta2": (H,)}

    def set_params(self, layer: int, params: dict) -> None:
        """params: name -> float32 array (bf16-exact values for bf16 slices)."""
        bufs = []
        for name in PARAM_NAMES:
            a = np.ascontiguousarray(params[name], dtype=np.float32)
            assert a.shape == self.shapes()[name], (name, a.shape)
            bufs.append(to_bf16_bits(a) if self.dtype == "bf16" else a)
        arr = (C.c_void_p * 12)(*[b.ctypes.data for b in bufs])
        L.call("sky_slice_set_params", self.h, layer, arr, 0)

    def _get(self, fn: str, layer: int, fp32: bool) -> dict:
        out = {}
        bufs = []
        for name in PARAM_NAMES:
            shp = self.shapes()[name]
            b = np.empty(shp, dtype=np.float32 if fp32 or self.dtype == "fp32" else np.uint16)
            bufs.append(b)
        arr = (C.c_void_p * 12)(*[b.ctypes.data for b in bufs])
        L.call(fn, self.h, layer, arr, 0)
        for name, b in zip(PARAM_NAMES, bufs):
            out[name] = from_bf16_bits(b) if b.dtype == np.uint16 else b
        return out

    def get_params(self, layer: int) -> dict:
        return self._get("sky_slice_get_params", layer, False)

    def get_grads(self, layer: int) -> dict:
        """fp32 gradients of the 12 tensors of `layer` from the last backward."""
        return self._get("sky_slice_get_grads", layer, True)

    # ---------------------------------------------------- local update (Sec. III)
    def optimizer_init(self, kind: str = "adamw", lr: float = 1e-4, beta1: float = 0.9,
                       beta2: float = 0.999, eps: float = 1e-6, weight_decay: float = 0.01,
                       momentum: float = 0.9) -> None:
        """fp32 master weights and zeroed AdamW / SGD state (see sky_slice.h)."""
        k = {"adamw": L.SKY_OPT_ADAMW, "sgd": L.SKY_OPT_SGD}[kind]
        cfg = L.SkyOptimizerConfig(k, lr, beta1, beta2, eps, weight_decay, momentum)
        L.call("sky_slice_optimizer_init", self.h, C.byref(cfg))

    def optimizer_step(self, lr: float, stream=None) -> None:
        """One update from the gradients of the last backward."""
        L.call("sky_slice_optimizer_step", self.h, C.c_float(lr), _stream_ptr(stream))

    def optimizer_state(self, layer: int, which: int) -> dict:
        """fp32 master weights (0), first (1) or second (2) state of `layer`."""
        bufs = [np.empty(self.shapes()[n], dtype=np.float32) for n in PARAM_NAMES]
        arr = (C.c_void_p * 12)(*[b.ctypes.data for b in bufs])
        L.call("sky_slice_get_optimizer_state", self.h, layer, which, arr)
        return dict(zip(PARAM_NAMES, bufs))

    # -------------------------------------------------------------- compute
    def forward(self, x, lens, y=None, stream=None, slot: int = 0):
        """x: device [B, S, H] tensor (slice dtype); lens: device int32 [B].
        ``slot`` picks the activation stash (sky_slice_forward_slot)."""
        import torch
        B, S, H = x.shape
        assert H == self.H and x.is_contiguous() and lens.dtype == torch.int32
        if y is None:
            y = torch.empty_like(x)
        L.call("sky_slice_forward_slot", self.h, _ptr(x), _ptr(lens), B, S, _ptr(y), slot,
               _stream_ptr(stream))
        if not hasattr(self, "_fwd_keep") or not isinstance(self._fwd_keep, dict):
            self._fwd_keep = {}
        self._fwd_keep[slot] = (x, lens)
        return y

    def backward(self, dy, dx=None, stream=None, slot: int = 0, accumulate: bool = False):
        """Backward of the last forward into ``slot``; ``accumulate`` adds the
        gradients to the current ones instead of overwriting them."""
        import torch
        if dx is None:
            dx = torch.empty_like(dy)
        L.call("sky_slice_backward_slot", self.h, _ptr(dy), _ptr(dx), slot, 1 if accumulate else 0,
               _stream_ptr(stream))
        return dx

    def step_graph(self, x, lens, y, dy, dx, stream=None) -> None:
        """Captures forward(x, lens, y) + backward(dy, dx) as one CUDA graph held
        by the slice (after running the step once); replay it with
        ``launch_step_graph``.  The five tensors stay bound to the graph."""
        import torch
        B, S, H = x.shape
        assert H == self.H and x.is_contiguous() and lens.dtype == torch.int32
        L.call("sky_slice_step_graph_create", self.h, _ptr(x), _ptr(lens), B, S, _ptr(y),
               _ptr(dy), _ptr(dx), _stream_ptr(stream))
        self._graph_keep = (x, lens, y, dy, dx)

    def launch_step_graph(self, stream=None) -> None:
        L.call("sky_slice_step_graph_launch", self.h, _stream_ptr(stream))

    def sync(self) -> None:
        L.call("sky_slice_sync", self.h)

    def layer_cost(self, B: int, S: int, iters: int = 5, lens=None) -> list:
        """Per-layer cost records (sky_slice_layer_cost).  ``lens``: the valid
        length of each of the B sequences (host ints); None = full length."""
        n = self.layer_end - self.layer_begin
        out = (L.SkyLayerCost * n)()
        lp = None
        if lens is not None:
            la = np.ascontiguousarray(lens, dtype=np.int32)
            assert la.shape == (B,)
            lp = la.ctypes.data_as(C.POINTER(C.c_int32))
        L.call("sky_slice_layer_cost", self.h, B, S, lp, iters, out, n)
        return [{f: getattr(o, f) for f, _ in L.SkyLayerCost._fields_ if f != "_pad"} for o in out]

    def set_profiling(self, on: bool) -> None:
        L.call("sky_slice_set_profiling", self.h, 1 if on else 0)

    def kernel_stats(self) -> dict:
        out = (L.SkyKernelStat * 16)()
        n = C.c_int32()
        L.call("sky_slice_kernel_stats", self.h, out, 16, C.byref(n))
        return {o.name.decode(): dict(launches=o.launches, total_ms=o.total_ms, flops=o.flops,
                                      bytes=o.bytes) for o in out[: n.value]}

    def memory(self) -> dict:
        v = [C.c_uint64() for _ in range(4)]
        L.call("sky_slice_memory", self.h, *[C.byref(x) for x in v])
        return dict(zip(("param_bytes", "grad_bytes", "stash_bytes", "workspace_bytes"),
                        [x.value for x in v]))

    def close(self) -> None:
        if getattr(self, "h", None):
            L.lib().sky_slice_destroy(self.h)
            self.h = None

    def __enter__(self):
        return self

    def __exit__(self, *a):
        self.close()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
