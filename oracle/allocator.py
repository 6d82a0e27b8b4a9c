"""Plain-Python oracle of the Sky Computing layer allocator (Sec. IV).

TEST INFRASTRUCTURE ONLY.  Nothing in the library's product path imports,
links or calls this module; only the tests do.  It shares no code with the
C++ allocator (``csrc/allocator.cpp``).

Problem (Sec. IV-C).  L layers, D devices.  Device ``i`` has a benchmark time
ratio ``dt[i]``, available memory ``dm[i]`` and communication time ``ct[i]``;
layer ``j`` has ``lf[j]`` FLOPs and needs ``lm[j]`` memory.  A partition index
``pi`` of length D+1 (Sec. IV-D) gives device ``i`` the layers
``pi[i] .. pi[i+1]-1``; ``pi[0] = 0`` and ``pi[D] = L``.

Functions, each following the passage named in its docstring:

* ``even_partition``          -- Sec. IV-A, equal layer counts.
* ``coarse_allocation``       -- Alg. 1, memory-driven boundary moves.
* ``finetune``                -- Alg. 2, workload-driven boundary moves.
* ``heuristic``               -- Alg. 1 followed by Alg. 2 (Sec. IV-D).
* ``milp_objective`` / ``milp_brute_force`` -- the mixed-integer model of
  Sec. IV-C, solved by enumerating every assignment (tiny instances only).

Readings of the paper where it is silent or inconsistent:

1. Workload.  Sec. IV-C writes ``w_i = dt_i * sum_j x_ij lf_j + ct_i`` (``ct``
   once per device); the text before Alg. 2 defines a layer's workload on
   device ``i`` as ``dt[i] * lf[j] + ct[i]`` and a device's workload as the sum
   over its layers (``ct`` once per layer).  Alg. 2 here uses the latter, as
   its own text says; the MILP objective uses the former, as the model says.
2. Even partition with ``L % D != 0``: the first ``L % D`` devices get one
   extra layer.
3. Alg. 1 compares against the memory of the next device's first layer,
   ``lm[pi[i+1]]``, and loops while ``dm[i] > am[i] + lm[pi[i+1]]`` (strict).
4. Alg. 2 recomputes device workloads from the current ``pi`` at every test
   (a move at boundary ``i`` is visible when boundary ``i+1`` is examined);
   the target (mean workload over all D devices) is computed once per sweep;
   "memory satisfied after change" means every device is within its memory
   after the move (only the two devices it touches can change).
5. Alg. 2 stops after a sweep that changes nothing, or after ``max_iter``
   sweeps.  (Its inner test ``counter == max_iter`` can never hold inside
   ``while counter < max_iter``; the loop bound is what limits the sweeps.)
6. The MILP leaves device order free and lets a device hold no layer (an
   empty device still contributes ``ct_i`` to ``q``, as the constraint reads).
7. Every sum (a device's memory or workload, the total workload) is
   accumulated left to right in index order (``_sum``), so the comparisons
   that decide a move round the same way wherever they are evaluated
   (Python's built-in ``sum`` compensates rounding from 3.12 on).
"""
from __future__ import annotations

import itertools


def _sum(values) -> float:
    """Plain left-to-right accumulation (reading 7)."""
    s = 0.0
    for v in values:
        s += v
    return s


def even_partition(L: int, D: int) -> list:
    """Sec. IV-A: an equal number of layers per device (reading 2)."""
    if D < 1 or L < D:
        raise ValueError("need 1 <= D <= L")
    base, extra = divmod(L, D)
    pi = [0]
    for i in range(D):
        pi.append(pi[-1] + base + (1 if i < extra else 0))
    return pi


def num_layers(pi: list, i: int) -> int:
    return pi[i + 1] - pi[i]


def allocated_memory(lm: list, pi: list) -> list:
    """``am[i]``: memory of the layers device ``i`` holds (Alg. 1)."""
    return [_sum(lm[pi[i]:pi[i + 1]]) for i in range(len(pi) - 1)]


def memory_satisfied(dm: list, lm: list, pi: list) -> bool:
    am = allocated_memory(lm, pi)
    return all(am[i] <= dm[i] for i in range(len(dm)))


def coarse_allocation(dm: list, lm: list, pi: list | None = None) -> list:
    """Alg. 1 (coarse allocation by memory).

    Starting from the even partition, every sweep visits boundaries
    ``i = 0 .. D-2``: while device ``i`` exceeds its memory and holds more
    than one layer it gives its last layer to device ``i+1``; then, while the
    next device's first layer fits on device ``i`` and device ``i+1`` keeps at
    least one layer, device ``i`` takes it.  Returns once every device fits;
    raises ``RuntimeError`` when a sweep changes nothing (reading 3)."""
    D, L = len(dm), len(lm)
    pi = list(pi) if pi is not None else even_partition(L, D)
    while True:
        if memory_satisfied(dm, lm, pi):
            return pi
        before = list(pi)
        for i in range(D - 1):
            am = allocated_memory(lm, pi)
            while am[i] > dm[i] and num_layers(pi, i) > 1:
                pi[i + 1] -= 1
                am = allocated_memory(lm, pi)
            while dm[i] > am[i] + lm[pi[i + 1]] and num_layers(pi, i + 1) > 1:
                pi[i + 1] += 1
                am = allocated_memory(lm, pi)
        if pi == before:
            raise RuntimeError("cannot fulfil the memory requirement")


def layer_workload(dt: list, lf: list, ct: list, i: int, j: int) -> float:
    """Workload of layer ``j`` on device ``i``: ``dt[i] * lf[j] + ct[i]`` (text before Alg. 2)."""
    return dt[i] * lf[j] + ct[i]


def device_workload(dt: list, lf: list, ct: list, pi: list, i: int) -> float:
    """Sum of the layer workloads of device ``i`` (reading 1)."""
    return _sum(layer_workload(dt, lf, ct, i, j) for j in range(pi[i], pi[i + 1]))


def finetune(dt: list, dm: list, ct: list, lf: list, lm: list, pi: list, max_iter: int) -> list:
    """Alg. 2 (optimise workload), readings 1, 4 and 5.

    Per sweep, target = mean device workload.  At boundary ``i``: if device
    ``i`` is below target, device ``i+1`` keeps a layer after the move and
    memory allows, device ``i`` takes device ``i+1``'s first layer; otherwise,
    if device ``i+1`` is below target, device ``i`` minus its last layer is
    still above target, device ``i`` keeps a layer and memory allows, device
    ``i`` gives its last layer to device ``i+1``."""
    D = len(dt)
    pi = list(pi)
    counter = 0
    while counter < max_iter:
        target = _sum(device_workload(dt, lf, ct, pi, i) for i in range(D)) / D
        before = list(pi)
        for i in range(D - 1):
            w_this = device_workload(dt, lf, ct, pi, i)
            take = list(pi)
            take[i + 1] += 1
            if w_this < target and num_layers(pi, i + 1) > 1 and memory_satisfied(dm, lm, take):
                pi = take
                continue
            w_next = device_workload(dt, lf, ct, pi, i + 1)
            w_last = layer_workload(dt, lf, ct, i, pi[i + 1] - 1)
            give = list(pi)
            give[i + 1] -= 1
            if (w_next < target and w_this - w_last > target and num_layers(pi, i) > 1
                    and memory_satisfied(dm, lm, give)):
                pi = give
        if pi == before:
            return pi
        counter += 1
    return pi


def heuristic(dt: list, dm: list, ct: list, lf: list, lm: list, max_iter: int = 100) -> list:
    """Sec. IV-D: coarse allocation (Alg. 1), then workload fine-tuning (Alg. 2)."""
    return finetune(dt, dm, ct, lf, lm, coarse_allocation(dm, lm), max_iter)


def milp_objective(dt: list, ct: list, lf: list, owner: list) -> float:
    """``q = max_i (dt_i * sum_j x_ij lf_j + ct_i)`` of Sec. IV-C for the
    assignment ``owner[j] = i`` (``x_ij = 1``)."""
    D = len(dt)
    return max(dt[i] * _sum(lf[j] for j in range(len(lf)) if owner[j] == i) + ct[i]
               for i in range(D))


def partition_owner(pi: list) -> list:
    """The MILP assignment of a partition index: layer ``j`` -> its device."""
    return [i for i in range(len(pi) - 1) for _ in range(pi[i], pi[i + 1])]


def milp_brute_force(dt: list, dm: list, ct: list, lf: list, lm: list):
    """Exact solution of the Sec. IV-C model by enumeration (reading 6).

    Every map of layers to devices is tried; a device's layers must be
    contiguous (``y_i - z_i = sum_j x_ij - 1``), each layer has one device and
    each device's layers fit its memory.  Returns ``(q, owner)`` of a minimum,
    or ``(inf, None)`` when nothing is feasible.  Only for tiny ``D ** L``."""
    D, L = len(dt), len(lf)
    best_q, best = float("inf"), None
    for owner in itertools.product(range(D), repeat=L):
        ok = True
        for i in range(D):
            idx = [j for j in range(L) if owner[j] == i]
            if idx and idx[-1] - idx[0] != len(idx) - 1:
                ok = False
                break
            if _sum(lm[j] for j in idx) > dm[i]:
                ok = False
                break
        if not ok:
            continue
        q = milp_objective(dt, ct, lf, list(owner))
        if q < best_q:
            best_q, best = q, list(owner)
    return best_q, best
