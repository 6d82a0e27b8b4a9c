"""Host logic of bench.py without a GPU: the timed region's barrier and
max-over-ranks reduction with two gloo ranks, and the FLOP accounting."""
import os
import socket
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402
from paper_2202_11836_gb300 import synth  # noqa: E402


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    import time
    import torch
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    counter = {"n": 0}

    def step():
        counter["n"] += 1
        time.sleep(0.002 * (rank + 1))

    t = {}

    def start():
        t["a"] = time.perf_counter()

    def stop():
        return (time.perf_counter() - t["a"]) * 1e3

    def reduce_max(v):
        x = torch.tensor([v], dtype=torch.float64)
        dist.all_reduce(x, op=dist.ReduceOp.MAX)
        return float(x.item())

    ms = bench.timed_region(step, 10, 3, lambda: None, dist.barrier, reduce_max, start, stop)
    out.put((rank, ms, counter["n"]))
    dist.destroy_process_group()


def test_timed_region_two_gloo_ranks():
    torch = pytest.importorskip("torch")
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    (r0, ms0, n0), (r1, ms1, n1) = res
    assert n0 == n1 == 13                 # warmup + timed steps on every rank
    assert ms0 == ms1                     # both ranks report the max
    assert ms0 >= 10 * 2 * 2.0 * 0.9      # the slower rank (4 ms per step) sets it


def test_flop_accounting_matches_closed_form():
    w = synth.WORKLOADS["large-s512"]
    lens = synth.lengths(w)
    g, a = bench.algorithmic_flops(w, lens)
    T, H, F = 8192, 1024, 4096
    assert g == 8 * 6 * T * (4 * H * H + 2 * H * F)
    assert a == 8 * 12 * H * 512 * int(lens.sum())
    # 80.2 M flop per token per layer at the mean valid length 384 of U{256..512}
    mean_len = (g + 8 * 12 * H * 512 * 16 * 384) / 8 / T
    assert abs(mean_len / 1e6 - 80.2) < 0.1


def test_gemm_shapes_cover_one_layer():
    """The per-shape GEMM table holds the 12 GEMMs of one layer (forward, data
    and weight gradients), whose FLOPs add up to 6 T (4 H^2 + 2 H F)."""
    import bench
    from paper_2202_11836_gb300 import synth
    w = synth.WORKLOADS["large-s512"]
    shapes = [s for s in bench.gemm_shapes(w) if not s[0].startswith("plain")]
    assert len(shapes) == 12
    T, H, F = w.tokens, w.hidden, w.ffn
    assert sum(2 * M * N * K for _, _, M, N, K, *_ in shapes) == 6 * T * (4 * H * H + 2 * H * F)


def test_allocation_plan_on_synthetic_layer_costs():
    """The bench's allocation object runs the host allocator (no GPU) on a
    160-layer table built from per-layer records: the exact ordered optimum
    is no worse than the heuristic, and the heuristic no worse than the even
    split, for devices whose speeds differ as the paper's slow-down factors."""
    rec = [{"fwd_ms": 0.25, "bwd_ms": 0.45, "param_bytes": 14_000_000,
            "grad_bytes": 28_000_000, "stash_bytes": 300_000_000} for _ in range(8)]
    plan = bench.allocation_plan(rec)
    m = plan["makespan_ms"]
    assert plan["layers"] == 160 and plan["devices"] == 64
    assert plan["layer_ms"] == 0.7
    assert m["best_in_device_order"] <= m["heuristic"] + 1e-9 <= m["even"] + 2e-9
    assert m["heuristic"] < m["even"]
