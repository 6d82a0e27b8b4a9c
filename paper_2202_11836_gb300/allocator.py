"""Python binding of the layer allocator (include/sky_alloc.h, Sec. IV).

Argument marshalling only: every step runs in the C++ library
(``csrc/allocator.cpp``).  A partition index ``pi`` (length D+1) gives device
``i`` the layers ``pi[i] .. pi[i+1]-1`` (Sec. IV-D); each device's range is
what one ``EncoderSlice(layer_begin=pi[i], layer_end=pi[i+1])`` runs.
"""
from __future__ import annotations

import ctypes as C

from . import _lib as L


class Problem:
    """Device table (``dt``, ``dm``, ``ct``, length D) and layer table (``lf``,
    ``lm``, length L) of Sec. IV-B, held as C arrays for the calls below."""

    def __init__(self, dt, dm, ct, lf, lm):
        self.D, self.L = len(dt), len(lf)
        if not (len(dm) == len(ct) == self.D and len(lm) == self.L):
            raise ValueError("dt, dm, ct need D entries and lf, lm L entries")
        D = C.c_double
        self._arrays = [(D * len(a))(*map(float, a)) for a in (dt, dm, ct, lf, lm)]
        self.c = L.SkyAllocProblem(self.D, self.L, *self._arrays)

    def _pi(self, values=None):
        return (C.c_int32 * (self.D + 1))(*(values or []))

    def coarse(self) -> list:
        """Alg. 1: memory-driven partition from the even start."""
        pi = self._pi()
        L.call("sky_alloc_coarse", C.byref(self.c), pi)
        return list(pi)

    def finetune(self, pi, max_iter: int = 100):
        """Alg. 2 from partition ``pi``; returns (pi, sweeps run)."""
        buf, sweeps = self._pi(pi), C.c_int32()
        L.call("sky_alloc_finetune", C.byref(self.c), max_iter, buf, C.byref(sweeps))
        return list(buf), sweeps.value

    def heuristic(self, max_iter: int = 100) -> list:
        """Sec. IV-D: Alg. 1, then Alg. 2."""
        pi = self._pi()
        L.call("sky_alloc_heuristic", C.byref(self.c), max_iter, pi)
        return list(pi)

    def workloads(self, pi, ct_per_layer: bool = False) -> list:
        """Per-device workloads (ct once per device as in Sec. IV-C, or per layer as in Alg. 2)."""
        w = (C.c_double * self.D)()
        model = L.SKY_COST_CT_PER_LAYER if ct_per_layer else L.SKY_COST_CT_PER_DEVICE
        L.call("sky_alloc_workloads", C.byref(self.c), self._pi(pi), model, w)
        return list(w)

    def makespan(self, pi) -> float:
        """q of Sec. IV-C for partition ``pi``: the slowest device's workload."""
        return max(self.workloads(pi))

    def best_ordered(self):
        """Exact best partition in device order; returns (pi, q)."""
        pi, q = self._pi(), C.c_double()
        L.call("sky_alloc_best_ordered", C.byref(self.c), pi, C.byref(q))
        return list(pi), q.value

    def milp_exact(self):
        """The Sec. IV-C model solved exactly (D <= 8); returns (owner per layer, q)."""
        owner, q = (C.c_int32 * self.L)(), C.c_double()
        L.call("sky_alloc_milp_exact", C.byref(self.c), owner, C.byref(q))
        return list(owner), q.value


def even(layers: int, devices: int) -> list:
    """Sec. IV-A: equal layer counts (the first L % D devices take one more)."""
    pi = (C.c_int32 * (devices + 1))()
    L.call("sky_alloc_even", layers, devices, pi)
    return list(pi)


def layer_table(costs) -> tuple:
    """``lf`` and ``lm`` of Sec. IV-B from ``EncoderSlice.layer_cost`` records:
    FLOPs of a layer's forward and backward pass, and its parameter, gradient
    and activation-stash bytes."""
    lf = [r["fwd_flops"] + r["bwd_flops"] for r in costs]
    lm = [r["param_bytes"] + r["grad_bytes"] + r["stash_bytes"] for r in costs]
    return lf, lm
