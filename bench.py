"""Throughput of one encoder-slice training step (forward + backward) on GB300.

A step is one pass of the whole hot path over one batch: the forward pass of
every layer of the slice, then the backward pass in reverse order with all
weight and input gradients (the per-device unit of work of the paper's
layer-partitioned training, Sec. III / IV-D).  Default workload: BERT-large
width, 8 layers, S=512, B=16 (bf16, seeded synthetic inputs standing in for
the paper's MNLI batches).  The timed step is the slice's forward + backward
captured once as a CUDA graph (sky_slice_step_graph_create) and replayed;
direct forward / backward calls are timed beside it.

Prints one JSON line (rank 0).  `--impl reference` times the float64 CPU
oracle instead (the reference arm).  With torchrun (N > 1) every rank runs an
independent replica on its own GPU (the path has no data-path collective) and
the slowest rank's time is reported.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2202_11836_gb300 import synth  # noqa: E402

METRIC = "encoder-slice fwd+bwd tokens/sec on 1 GB300; % of bf16 tensor-core peak"
DEFAULT_WORKLOAD = "large-s512"
L2_BYTES = 129 * 2 ** 20


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return dict(hbm=d["hbm_gbs"], bf16=d["bf16_tflops"], bf16_sus=d["bf16_tflops_sustained"],
                    source="measured")
    return dict(hbm=6800.0, bf16=1900.0, bf16_sus=1700.0, source="fallback")


# DRAM traffic of the dominant kernel: dram__bytes_read.sum + dram__bytes_write.sum
# per gemm_tc_kernel launch, averaged over the 12 GEMM launches of one layer
# (layer 0 forward, layer 7 backward) in one ncu capture of the bench
# workload.  It describes the kernel sources it was taken on: when any of them
# changes (SHA-256 prefix below) the figure no longer applies and the bench
# reports null until a new capture replaces it.
GEMM_TRAFFIC = {
    "workload": "large-s512",
    "bytes_per_launch": 74.43e6,
    "sources": {"gemm_tc.cu": "751133252cea931d", "gemm.h": "04ea90b6fdc49866", "ptx.cuh": "f0b810e074f474e4", "common.cuh": "c40ceaff9f8d8dcd"},
}


def gemm_traffic(workload):
    """The recorded per-launch GEMM DRAM traffic, or None if it does not apply."""
    import hashlib
    if workload != GEMM_TRAFFIC["workload"]:
        return None
    csrc = os.path.join(ROOT, "paper_2202_11836_gb300", "csrc")
    for name, digest in GEMM_TRAFFIC["sources"].items():
        with open(os.path.join(csrc, name), "rb") as f:
            if hashlib.sha256(f.read()).hexdigest()[:16] != digest:
                return None
    return GEMM_TRAFFIC["bytes_per_launch"]


def allocation_plan(rec, layers=160, devices=64, seed=2022):
    """The paper's allocator on the measured layer costs (Sec. IV).

    The layer table is the median per-layer cost of the benchmark slice
    (time of fwd + bwd on this GPU, parameter + gradient + stash bytes),
    repeated for a 160-layer model; the device table has 64 devices whose time
    ratios are drawn like the paper's slow-down factors (normal, clipped to
    [1, 7]) and whose memory holds 1.5 to 4 times an even share.  Reports the
    predicted per-step makespan (slowest device, ms) of the even split, the
    heuristic (Alg. 1 + Alg. 2) and the exact best partition in device order,
    and the C++ heuristic's run time."""
    import random
    from paper_2202_11836_gb300 import allocator
    t_layer = statistics.median([r["fwd_ms"] + r["bwd_ms"] for r in rec])
    m_layer = float(statistics.median([r["param_bytes"] + r["grad_bytes"] + r["stash_bytes"]
                                       for r in rec]))
    rng = random.Random(seed)
    dt = [min(7.0, max(1.0, rng.gauss(4.0, 1.5))) for _ in range(devices)]
    share = m_layer * layers / devices
    dm = [rng.uniform(1.5, 4.0) * share for _ in range(devices)]
    P = allocator.Problem(dt, dm, [0.0] * devices, [t_layer] * layers, [m_layer] * layers)
    t0 = time.perf_counter()
    pi = P.heuristic(100)
    t_heur = (time.perf_counter() - t0) * 1e3
    _, q_best = P.best_ordered()
    return {"layers": layers, "devices": devices, "layer_ms": round(t_layer, 4),
            "makespan_ms": {"even": round(P.makespan(allocator.even(layers, devices)), 3),
                            "heuristic": round(P.makespan(pi), 3),
                            "best_in_device_order": round(q_best, 3)},
            "heuristic_run_ms": round(t_heur, 3)}


def algorithmic_flops(w, lens):
    """Matmul FLOPs of one step (forward + backward) over all layers."""
    T, H, F, S = w.batch * w.seq, w.hidden, w.ffn, w.seq
    gemm = 3 * 2 * T * (4 * H * H + 2 * H * F)
    attn = 3 * 4 * H * S * int(np.sum(lens))
    return w.layers * gemm, w.layers * attn


# ----------------------------------------------------------------- clocks
class ClockSampler:
    """Samples nvidia-smi clocks and throttle reasons while the timed region runs."""
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id: str):
        self.idx = gpu_id
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100", "-i", str(self.idx)], stdout=subprocess.PIPE,
                stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except (OSError, FileNotFoundError):
            self.proc = None
        time.sleep(0.3)
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *a):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for l in self.lines:
            f = [x.strip() for x in l.split(",")]
            if len(f) < 8:
                continue
            try:
                sm.append(float(f[0])); mx.append(float(f[1]))
            except ValueError:
                continue
            for n, v in zip(names, f[4:8]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


# ------------------------------------------------------------ distributed
def dist_env():
    return int(os.environ.get("RANK", 0)), int(os.environ.get("WORLD_SIZE", 1)), \
        int(os.environ.get("LOCAL_RANK", 0))


def timed_region(step, steps, warmup, sync, barrier, reduce_max, start_event, stop_event):
    """W untimed steps, then K steps between a barrier + sync on both sides.

    Returns the slowest rank's elapsed milliseconds for the K steps."""
    for _ in range(warmup):
        step()
    sync()
    barrier()
    sync()
    start_event()
    for _ in range(steps):
        step()
    ms = stop_event()
    sync()
    barrier()
    return reduce_max(ms)


# ------------------------------------------------------------- CPU oracle
def oracle_sample(w, seconds: float):
    """Times the float64 oracle on one sequence and one layer of workload ``w``
    (forward + backward) until ``seconds`` have passed; returns tokens/s of
    the whole slice and a description."""
    from oracle import encoder_f64 as ORC
    lens = synth.lengths(w)
    b = int(np.argmax(lens))
    X = synth.activations(w, batch=b + 1)[b:b + 1].astype(np.float64)
    dY = synth.upstream_grad(w, batch=b + 1)[b:b + 1].astype(np.float64)
    p = synth.layer_params(w.layer_begin, w.hidden, w.ffn, w.dtype)
    p = {k: v.astype(np.float64) for k, v in p.items()}
    n, t0 = 0, time.perf_counter()
    while True:
        ORC.slice_step(X, lens[b:b + 1], dY, [p], w.heads, 1e-12)
        n += 1
        el = time.perf_counter() - t0
        if el >= seconds:
            break
    per_layer_seq = el / n
    tok_s = w.seq / (per_layer_seq * w.layers)
    desc = (f"{n} x (1 sequence of S={w.seq} (len {int(lens[b])}), 1 of {w.layers} layers, fwd+bwd,"
            f" float64 numpy) in {el:.1f} s; scaled to the {w.layers}-layer slice")
    return tok_s, desc, per_layer_seq


def cpu_cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count()


def run_reference(args, w):
    """The reference arm: the float64 oracle on the host cores.  One "step"
    here is what is timed, a bounded sample of the workload (one sequence x
    one layer, forward + backward); ``ms_per_step`` and ``steps`` describe
    those samples, and ``value`` scales the median sample time to the whole
    slice's tokens/s by the factor stated in ``sample_scale``."""
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    from oracle import encoder_f64 as ORC  # noqa: F401
    for _ in range(args.warmup):
        oracle_sample(w, 0.0)
    vals, times = [], []
    for _ in range(args.steps):
        v, desc, t = oracle_sample(w, 0.0)
        vals.append(v); times.append(t)
    value = statistics.median(vals)
    ms = statistics.median(times) * 1e3
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": ms, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "f64", "data": "synthetic", "config": config_of(w),
            "sample_scale": {"step_is": "1 sequence x 1 layer, forward + backward",
                             "tokens_per_sample": w.seq, "samples_per_full_step": w.layers * w.batch,
                             "full_step_ms_estimate": ms * w.layers * w.batch,
                             "value_is": "tokens_per_step / (ms_per_step x samples_per_full_step)"},
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": cpu_cores(),
                             "kind": "oracle",
                             "sample": "each step: 1 sequence x 1 layer fwd+bwd of the workload, "
                                       "scaled to the whole slice"},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def config_of(w):
    return {"workload": w.name, "layers": w.layers, "hidden": w.hidden, "heads": w.heads,
            "ffn": w.ffn, "seq": w.seq, "batch": w.batch, "tokens_per_step": w.tokens,
            "dtype": w.dtype, "l2": "inputs larger than L2 (the step streams a multi-GB "
            "activation stash; no explicit flush)"}


# ---------------------------------------------------------------- GPU arm
def run_gpu(args, w):
    import torch
    import torch.distributed as dist
    from paper_2202_11836_gb300 import _lib
    from paper_2202_11836_gb300.slice import EncoderSlice

    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    dev = torch.device("cuda", local)

    lens = synth.lengths(w)
    s = EncoderSlice(w.hidden, w.heads, w.ffn, w.layer_begin, w.layer_begin + w.layers,
                     w.batch, w.seq, w.dtype)
    for l in range(w.layer_begin, w.layer_begin + w.layers):
        s.set_params(l, synth.layer_params(l, w.hidden, w.ffn, w.dtype))
    tdt = torch.bfloat16 if w.dtype == "bf16" else torch.float32
    X = synth.activations(w)
    dY = synth.upstream_grad(w)
    x = torch.from_numpy(X).to(dev).to(tdt)
    dy = torch.from_numpy(dY).to(dev).to(tdt)
    ln = torch.from_numpy(lens).to(dev)
    y = torch.empty_like(x)
    dx = torch.empty_like(x)
    stream = torch.cuda.current_stream(dev)

    def step():
        s.forward(x, ln, y, stream)
        s.backward(dy, dx, stream)

    # the same step captured once as a CUDA graph held by the slice
    # (sky_slice_step_graph_create); replays launch the same kernels
    s.step_graph(x, ln, y, dy, dx, stream)

    def step_graph():
        s.launch_step_graph(stream)

    def barrier():
        if world > 1:
            dist.barrier()

    def reduce_max(v):
        if world > 1:
            t = torch.tensor([v], dtype=torch.float64, device=dev)
            dist.all_reduce(t, op=dist.ReduceOp.MAX)
            return float(t.item())
        return v

    ev = {}

    def start():
        ev["a"] = torch.cuda.Event(enable_timing=True)
        ev["b"] = torch.cuda.Event(enable_timing=True)
        ev["a"].record(stream)

    def stop():
        ev["b"].record(stream)
        ev["b"].synchronize()
        return ev["a"].elapsed_time(ev["b"])

    sync = torch.cuda.synchronize
    # 1. device-resident throughput
    launches0 = _lib.lib().sky_launch_count()
    props = torch.cuda.get_device_properties(local)
    gpu_id = ("GPU-" + str(props.uuid)) if getattr(props, "uuid", None) else str(local)
    with ClockSampler(gpu_id) as clk:
        ms = timed_region(step_graph, args.steps, args.warmup, sync, barrier, reduce_max, start,
                          stop)
    launches = (_lib.lib().sky_launch_count() - launches0)
    launches_timed = launches * args.steps // (args.steps + args.warmup)
    s.sync()
    # 1b. the same replayed step over a seconds-long region, so the clock
    # record covers a sustained run (read against the sustained peak)
    sustained = None
    if args.sustain_s > 0:
        n_sus = max(args.steps, int(round(args.sustain_s / (ms / args.steps / 1e3))))
        with ClockSampler(gpu_id) as clk_sus:
            ms_sus = timed_region(step_graph, n_sus, 3, sync, barrier, reduce_max, start, stop)
        s.sync()
        sus_flops = sum(algorithmic_flops(w, lens))
        sustained = {"steps": n_sus, "seconds": round(ms_sus / 1e3, 3),
                     "ms_per_step": ms_sus / n_sus,
                     "value": world * w.tokens * n_sus / (ms_sus / 1e3),
                     "pct_bf16_peak_sustained": round(100 * sus_flops / (ms_sus / n_sus / 1e3)
                                                      / 1e12 / peaks()["bf16_sus"], 2),
                     "pct_bf16_peak_burst": round(100 * sus_flops / (ms_sus / n_sus / 1e3)
                                                  / 1e12 / peaks()["bf16"], 2),
                     "clocks": clk_sus.summary()}
    # the same steps as direct sky_slice_forward / sky_slice_backward calls
    ms_direct = timed_region(step, args.steps, args.warmup, sync, barrier, reduce_max, start, stop)
    s.sync()
    ms_step = ms / args.steps
    tokens = w.tokens
    value = world * tokens * args.steps / (ms / 1e3)
    gemm_flops, attn_flops = algorithmic_flops(w, lens)
    pk = peaks()

    # 2. per-kernel CUDA-event timing of the same steps (roofline of the
    # dominant kernel): every kernel in line on the caller's stream between a
    # pair of events.  (The same timers captured into the step graph and
    # replayed, sky_slice_step_graph_create with profiling on, read about 2%
    # slower per GEMM: the event nodes serialise the graph as well.)
    s.set_profiling(True)
    timed_region(step, max(3, args.steps // 4), 1, sync, barrier, reduce_max, start, stop)
    stats = s.kernel_stats()
    s.set_profiling(False)
    gemm_ms = sum(v["total_ms"] for k, v in stats.items() if k.startswith("gemm"))
    gemm_f = sum(v["flops"] for k, v in stats.items() if k.startswith("gemm"))
    gemm_n = sum(v["launches"] for k, v in stats.items() if k.startswith("gemm"))
    achieved = gemm_f / (gemm_ms / 1e3) / 1e12 if gemm_ms > 0 else 0.0
    kernel_table = {k: {"launches": v["launches"], "ms": round(v["total_ms"], 4),
                        "share": round(v["total_ms"] / max(1e-9, sum(x["total_ms"] for x in stats.values())), 4),
                        "tflops": round(v["flops"] / (v["total_ms"] / 1e3) / 1e12, 1) if v["flops"] else None,
                        "gbs": round(v["bytes"] / (v["total_ms"] / 1e3) / 1e9, 1) if v["bytes"] else None}
                    for k, v in stats.items()}

    # 3. per-layer cost (the allocator's per-layer time) on the workload's own lengths
    rec = s.layer_cost(w.batch, w.seq, iters=5, lens=lens)
    per_layer_ms = statistics.median([r["fwd_ms"] + r["bwd_ms"] for r in rec])
    per_layer_flops = statistics.median([r["fwd_flops"] + r["bwd_flops"] for r in rec])

    # 3b. the local parameter update (Sec. III), timed on its own: AdamW over
    # every parameter of the slice, an HBM stream of 20-30 bytes per parameter
    s.optimizer_init(args.optimizer, lr=2e-5, beta1=0.9, beta2=0.999, eps=1e-6, weight_decay=0.01)
    n_params = sum(int(np.prod(v)) for v in s.shapes().values()) * w.layers
    for _ in range(3):
        s.optimizer_step(2e-5, stream)
    sync()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    n_upd = 10
    t0.record(stream)
    for _ in range(n_upd):
        s.optimizer_step(2e-5, stream)
    t1.record(stream)
    t1.synchronize()
    upd_ms = t0.elapsed_time(t1) / n_upd
    # bytes per parameter: AdamW reads g, w, m, v and writes w, m, v (and, in a
    # bf16 slice, the parameter rounded to bf16); SGD reads g, w, b and writes
    # w, b (and the bf16 parameter).  An fp32 slice updates its parameters in place.
    bpp = (30 if args.optimizer == "adamw" else 22) if w.dtype == "bf16" else \
        (28 if args.optimizer == "adamw" else 20)
    upd_gbs = bpp * n_params / (upd_ms / 1e3) / 1e9
    optimizer = {"kind": args.optimizer, "params": n_params, "ms": round(upd_ms, 4),
                 "bytes_per_param": bpp, "achieved_gbs": round(upd_gbs, 1),
                 "peak_gbs": pk["hbm"], "frac": round(upd_gbs / pk["hbm"], 4)}

    # 4. end to end through the public API with host buffers
    xh = torch.from_numpy(X).to(tdt).pin_memory()
    dyh = torch.from_numpy(dY).to(tdt).pin_memory()
    lh = torch.from_numpy(lens).pin_memory()
    yh = torch.empty_like(xh).pin_memory()
    dxh = torch.empty_like(xh).pin_memory()
    h2d = xh.numel() * xh.element_size() * 2 + lh.numel() * 4
    d2h = yh.numel() * yh.element_size() * 2

    # The host copies run on a copy stream, pipelined with the compute: a
    # step's inputs are copied to device staging buffers while the previous
    # step computes, and its results are copied back while the next one
    # computes.  On the compute stream each step moves its inputs from the
    # staging buffers into the graph's buffers and its results out to the
    # output staging buffers (device-to-device, inside the step).  Every
    # step still carries one host-to-device copy of its inputs and one
    # device-to-host copy of its results, all inside the timed region but
    # the first step's input copy (made during the last untimed step); the
    # region ends when the last step's results have reached the host.
    copy_st = torch.cuda.Stream(device=dev)
    xs, dys, lns = torch.empty_like(x), torch.empty_like(dy), torch.empty_like(ln)
    ys, dxs = torch.empty_like(y), torch.empty_like(dx)
    ev_h2d, ev_in_free = torch.cuda.Event(), torch.cuda.Event()
    ev_out, ev_d2h = torch.cuda.Event(), torch.cuda.Event()

    def h2d_after(ev):  # next inputs -> staging, once the staging buffers are free
        with torch.cuda.stream(copy_st):
            if ev is not None:
                copy_st.wait_event(ev)
            xs.copy_(xh, non_blocking=True)
            dys.copy_(dyh, non_blocking=True)
            lns.copy_(lh, non_blocking=True)
            ev_h2d.record(copy_st)

    h2d_after(None)
    ev_d2h.record(copy_st)

    def step_e2e():
        stream.wait_event(ev_h2d)
        x.copy_(xs, non_blocking=True)
        dy.copy_(dys, non_blocking=True)
        ln.copy_(lns, non_blocking=True)
        ev_in_free.record(stream)
        h2d_after(ev_in_free)
        s.launch_step_graph(stream)
        stream.wait_event(ev_d2h)  # the previous results have left the staging buffers
        ys.copy_(y, non_blocking=True)
        dxs.copy_(dx, non_blocking=True)
        ev_out.record(stream)
        with torch.cuda.stream(copy_st):
            copy_st.wait_event(ev_out)
            yh.copy_(ys, non_blocking=True)
            dxh.copy_(dxs, non_blocking=True)
            ev_d2h.record(copy_st)

    def stop_e2e():
        stream.wait_event(ev_d2h)  # the last step's results are on the host
        return stop()

    ms_e2e = timed_region(step_e2e, args.steps, 2, sync, barrier, reduce_max, start, stop_e2e)
    e2e_value = world * tokens * args.steps / (ms_e2e / 1e3)
    s.sync()

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu:
        v, desc, _ = oracle_sample(w, args.cpu_seconds)
        cpu = {"value": v, "unit": "tokens/s", "cores": cpu_cores(), "kind": "oracle",
               "sample": desc}

    if rank == 0:
        total_f = gemm_flops + attn_flops
        line = {
            "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_step,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": w.dtype,
            "data": "synthetic", "config": config_of(w),
            "pct_bf16_peak_end_to_end": round(100 * total_f / (ms_step / 1e3) / 1e12 / pk["bf16"], 2),
            "tokens_per_s_per_layer": tokens / (per_layer_ms / 1e3),
            "per_layer_ms": per_layer_ms,
            "per_layer": {"ms": per_layer_ms, "lengths": "the workload's own (same mask as value)",
                          "pct_bf16_peak": round(100 * per_layer_flops / (per_layer_ms / 1e3)
                                                 / 1e12 / pk["bf16"], 2),
                          "how": "sky_slice_layer_cost: median over layers of fwd+bwd; CUDA "
                                 "events per layer, captured with one pass into a graph and "
                                 "replayed (per-layer times add up to the pass)"},
            "allocation": allocation_plan(rec),
            "optimizer": optimizer,
            "valid_tokens_per_s": world * int(np.sum(lens)) * args.steps / (ms / 1e3),
            "step": "one CUDA graph of the slice's forward + backward (sky_slice_step_graph_launch)",
            "sustained": sustained,
            "direct_calls": {"value": world * tokens * args.steps / (ms_direct / 1e3),
                             "ms_per_step": ms_direct / args.steps,
                             "how": "sky_slice_forward + sky_slice_backward each step"},
            "roofline": {"kernel": "gemm_tc_kernel (all GEMM launches of the step)",
                         "bound": "tensor", "achieved": round(achieved, 1),
                         "peak": pk["bf16"], "unit": "TFLOP/s",
                         "frac": round(achieved / pk["bf16"], 4),
                         "frac_of_sustained_peak": round(achieved / pk["bf16_sus"], 4),
                         "peak_source": pk["source"] + " (burst bf16: the per-kernel region is "
                                                       "a few steps long; sustained also given)",
                         "traffic": gemm_traffic(w.name), "traffic_unit": "bytes per launch",
                         "launches": gemm_n,
                         "timing": "CUDA events around every launch, all kernels in line on "
                                   "the caller's stream"},
            "kernels": kernel_table,
            "cpu_baseline": cpu,
            "e2e": {"value": e2e_value, "unit": "tokens/s", "h2d_bytes_per_step": h2d,
                    "d2h_bytes_per_step": d2h},
            "gpu_launches": int(launches_timed),
            "clocks": clk.summary(),
        }
        print(json.dumps(line), flush=True)
    s.close()
    if world > 1:
        dist.destroy_process_group()
    return 0


def gemm_shapes(w):
    """The 13 GEMMs of one encoder layer of workload ``w`` as sky_gemm calls:
    (name, form, M, N, K, epilogue, bias, fp32 output, aux in, aux out)."""
    T, H, F = w.tokens, w.hidden, w.ffn
    return [
        ("fwd QKV", "XWT", T, 3 * H, H, "STORE", True, False, None, None),
        ("fwd attn-out", "XWT", T, H, H, "STORE", True, True, None, None),
        ("fwd FFN1", "XWT", T, F, H, "BIAS_GELU", True, False, None, "f16"),
        ("fwd FFN2", "XWT", T, H, F, "STORE", True, True, None, None),
        ("dgrad FFN2", "XW", T, F, H, "GELU_BWD", False, False, "f16", None),
        ("dgrad FFN1", "XW", T, H, F, "STORE", False, True, None, None),
        ("dgrad attn-out", "XW", T, H, H, "STORE", False, False, None, None),
        ("dgrad QKV", "XW", T, H, 3 * H, "STORE", False, True, None, None),
        ("wgrad W2", "XTW", H, F, T, "STORE", False, True, None, None),
        ("wgrad W1", "XTW", F, H, T, "STORE", False, True, None, None),
        ("wgrad Wo", "XTW", H, H, T, "STORE", False, True, None, None),
        ("wgrad Wqkv", "XTW", 3 * H, H, T, "STORE", False, True, None, None),
        ("plain FFN1 shape", "XWT", T, F, H, "STORE", False, False, None, None),
    ]


def run_gemm_shapes(args, w):
    """Times every GEMM shape of one layer alone through sky_gemm (bf16 in,
    fp32 accumulation): L2 flushed by a 256 MB write before each launch,
    ``--warmup`` untimed and ``--steps`` timed launches per shape (CUDA events
    around each), median.  sky_gemm has no residual operand, so the two
    residual-branch forward GEMMs and two data gradients run without it.
    ``--only`` picks shapes by name (comma-separated substrings)."""
    import ctypes as C

    import torch
    from paper_2202_11836_gb300 import _lib as L

    def ptr(t):
        return C.c_void_p(0 if t is None else int(t.data_ptr()))

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    st = torch.cuda.current_stream(dev)
    sp = C.c_void_p(int(st.cuda_stream))
    gen = torch.Generator(device=dev).manual_seed(synth.SEED)
    flush = torch.empty(256 * 2 ** 20, dtype=torch.uint8, device=dev)
    forms = {"XWT": L.SKY_GEMM_XWT, "XW": L.SKY_GEMM_XW, "XTW": L.SKY_GEMM_XTW}
    epis = {"STORE": L.SKY_EPI_STORE, "BIAS_GELU": L.SKY_EPI_BIAS_GELU,
            "GELU_BWD": L.SKY_EPI_GELU_BWD}
    bf = L.SKY_DTYPE_BF16
    picks = [p for p in (args.only or "").split(",") if p]
    total_us, total_f, rows = 0.0, 0.0, []
    for name, form, M, N, K, epi, bias, f32, aux_in, aux_out in gemm_shapes(w):
        if picks and not any(p in name for p in picks):
            continue
        a_shape = (K, M) if form == "XTW" else (M, K)
        b_shape = (N, K) if form == "XWT" else (K, N)
        A = torch.randn(a_shape, device=dev, generator=gen).bfloat16()
        Bm = (0.02 * torch.randn(b_shape, device=dev, generator=gen)).bfloat16()
        Cm = torch.empty((M, N), device=dev, dtype=torch.float32 if f32 else torch.bfloat16)
        bv = torch.zeros(N, device=dev, dtype=torch.bfloat16) if bias else None
        ai = torch.rand((M, N), device=dev, generator=gen).half() if aux_in else None
        ao = torch.empty((M, N), device=dev, dtype=torch.float16) if aux_out else None
        odt = L.SKY_DTYPE_FP32 if f32 else bf
        wsb = L.lib().sky_gemm_workspace_bytes(forms[form], M, N, K, bf, odt)
        ws = torch.empty(max(wsb, 16), dtype=torch.uint8, device=dev)
        times = []
        for it in range(args.warmup + args.steps):
            flush.zero_()
            # a 50 us device-side wait after the flush, so that the GEMM is
            # already queued when e0 fires: the host's own call time stays
            # out of the measured interval
            L.call("sky_device_delay", 50000, sp)
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(st)
            L.call("sky_gemm", forms[form], M, N, K, bf, ptr(A), ptr(Bm), ptr(Cm), odt, epis[epi],
                   ptr(bv), ptr(ai), ptr(ao), ptr(ws), wsb, None, sp)
            e1.record(st)
            e1.synchronize()
            if it >= args.warmup:
                times.append(e0.elapsed_time(e1) * 1e3)
        us = statistics.median(times)
        f = 2.0 * M * N * K
        total_us += us
        total_f += f
        rows.append({"gemm": name, "M": M, "N": N, "K": K, "epilogue": epi, "fp32_out": f32,
                     "us": round(us, 2), "tflops": round(f / us / 1e6, 1)})
        print(f"{name:18s} M={M:6d} N={N:6d} K={K:6d} {epi:9s} f32={int(f32)} "
              f"{us:8.1f} us {f / us / 1e6:8.1f} TF/s", flush=True)
    if rows:
        print(f"TOTAL {total_us:.1f} us  {total_f / total_us / 1e6:.1f} TF/s", flush=True)
    print(json.dumps({"gemm_shapes": rows, "workload": w.name, "launches_timed": args.steps,
                      "l2": "flushed before each launch"}), flush=True)
    return 0


def run_uneven(args, w):
    """The load-balanced uneven slices of the 160-layer base-width model
    (lengths 1, 3, 7, 17; Sec. IV-D partitions), each run on its own: the
    per-slice step time (graph replays, CUDA events, ``--steps`` after
    ``--warmup``), the per-layer cost records of sky_slice_layer_cost, and a
    least-squares fit t(n) = alpha + beta n of slice time over layer count."""
    import torch
    from paper_2202_11836_gb300.slice import EncoderSlice

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    st = torch.cuda.current_stream(dev)
    lens = synth.lengths(w)
    x = torch.from_numpy(synth.activations(w)).to(dev).to(torch.bfloat16)
    dy = torch.from_numpy(synth.upstream_grad(w)).to(dev).to(torch.bfloat16)
    ln = torch.from_numpy(lens).to(dev)
    y, dx = torch.empty_like(x), torch.empty_like(x)
    rows = []
    for lb, le in synth.UNEVEN_SLICES:
        with EncoderSlice(w.hidden, w.heads, w.ffn, lb, le, w.batch, w.seq, "bf16") as s:
            for l in range(lb, le):
                s.set_params(l, synth.layer_params(l, w.hidden, w.ffn, "bf16"))
            s.step_graph(x, ln, y, dy, dx, st)
            for _ in range(args.warmup):
                s.launch_step_graph(st)
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            torch.cuda.synchronize()
            e0.record(st)
            for _ in range(args.steps):
                s.launch_step_graph(st)
            e1.record(st)
            e1.synchronize()
            ms = e0.elapsed_time(e1) / args.steps
            s.sync()
            rec = s.layer_cost(w.batch, w.seq, iters=5, lens=lens)
        layer_ms = [r["fwd_ms"] + r["bwd_ms"] for r in rec]
        rows.append({"layers": [lb, le], "n": le - lb, "ms_per_step": round(ms, 4),
                     "tokens_per_s": round(w.tokens / (ms / 1e3), 1),
                     "sum_layer_cost_ms": round(sum(layer_ms), 4),
                     "median_layer_cost_ms": round(statistics.median(layer_ms), 4)})
    n = np.array([r["n"] for r in rows], float)
    fits = {}
    for key in ("ms_per_step", "sum_layer_cost_ms"):
        t = np.array([r[key] for r in rows])
        beta, alpha = np.polyfit(n, t, 1)
        pred = alpha + beta * n
        r2 = 1.0 - float(((t - pred) ** 2).sum() / ((t - t.mean()) ** 2).sum())
        fits[key] = {"alpha_ms": round(float(alpha), 4), "beta_ms_per_layer": round(float(beta), 4),
                     "r2": round(r2, 6)}
    print(json.dumps({"workload": w.name, "slices": rows, "fit": fits,
                      "config": config_of(w)}), flush=True)
    return 0


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD, choices=sorted(synth.WORKLOADS))
    ap.add_argument("--cpu-seconds", type=float, default=10.0)
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--optimizer", default="adamw", choices=["adamw", "sgd"],
                    help="local update rule timed after the step")
    ap.add_argument("--sustain-s", type=float, default=2.0,
                    help="length of the second, sustained timed region (seconds; 0 = skip)")
    ap.add_argument("--gemm-shapes", action="store_true",
                    help="time each GEMM shape of one layer alone through sky_gemm")
    ap.add_argument("--uneven", action="store_true",
                    help="time the uneven slices {1,3,7,17} of the 160-layer base-width model")
    ap.add_argument("--only", default="", help="with --gemm-shapes: shapes whose name "
                    "contains one of these comma-separated strings")
    args = ap.parse_args(argv)
    assert args.warmup >= 0 and args.steps >= 1
    w = synth.WORKLOADS[args.workload]
    if args.impl == "reference":
        return run_reference(args, w)
    if args.gemm_shapes:
        return run_gemm_shapes(args, w)
    if args.uneven:
        return run_uneven(args, synth.WORKLOADS["base-s128-b16"])
    return run_gpu(args, w)


if __name__ == "__main__":
    sys.exit(main())
