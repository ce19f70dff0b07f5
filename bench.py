#!/usr/bin/env python3
"""Benchmark: one fwd+bwd adaptation step of 17 concurrent ViT-B V-MoE expert layers.

A step is the whole hot path -- route, dispatch, expert FFN forward, combine,
weighted dispatch of dY, expert FFN backward (dH, dX, dW1, dW2), combine of dX --
over one batch of synthetic tokens (T=17 tasks x 8 images x 197 tokens, d=768,
f=3072, E=32 experts per task, top-2, capacity factor 1.25, drifted router).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Prints ONE JSON line on rank 0.  ``value`` is tokens/s of the whole job with every
input resident in HBM (device-timed with CUDA events, max over ranks); ``e2e`` is
the same metric through the public API from pinned host buffers with the
host<->device copies inside the timed region.  ``--impl reference`` times the fp64
CPU oracle on a bounded sample of the same workload instead.

Multi-GPU (torchrun, one process per GPU): the step partitions by task, so every
rank runs its own 17-task workload with no data-path collective ("weak" scaling);
the process group only provides the barrier and the max over ranks of the time.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import workloads  # noqa: E402

METRIC = "expert-layer fwd+bwd tokens/sec at 17-task ViT-B V-MoE; % bf16 tensor peak"
UNIT = "tokens/s"
L2_NOTE = ("inputs larger than L2: every step streams the 5.1 GB of expert weights "
           "(plus 5.1 GB of weight gradients), 40x the 129 MB L2")


def load_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as fh:
            pk = json.load(fh)
        return dict(hbm_gbs=pk["hbm_gbs"], bf16_tflops=pk["bf16_tflops"],
                    bf16_tflops_sustained=pk.get("bf16_tflops_sustained", pk["bf16_tflops"]),
                    source="measured")
    except Exception:
        return dict(hbm_gbs=6800.0, bf16_tflops=1900.0, bf16_tflops_sustained=1700.0,
                    source="fallback")


# ----------------------------------------------------------------------------- byte / flop model
def model_counts(cfg, loads):
    """Algorithmic bytes and flops per launch of each kernel, from the actual loads.

    A = kept assignments, G = T*E groups, Gp = groups with load > 0; 2-byte elements
    for bf16 activations and weights.  Only bytes the definition must move count:
    kept rows, every weight of a non-empty group once, every output once.
    """
    T, N, d, f, E, k = cfg.T, cfg.N, cfg.d, cfg.f, cfg.E, cfg.k
    el = 2 if cfg.dtype == "bf16" else 4
    A = int(sum(loads))
    G = T * E
    Gp = int(sum(1 for v in loads if v > 0))
    C = cfg.capacity
    idx_bytes = T * N * k * 4
    w = Gp * d * f * el
    gemm_flops = 2.0 * A * d * f
    return {
        "route_topk": (T * N * d * el + T * d * E * 4 + T * E * 4 + T * N * E * 4 + 2 * idx_bytes, 2.0 * T * N * d * E),
        "capacity_scan": (2 * idx_bytes + T * E * 4, 0.0),
        "dispatch": (A * d * el + 2 * idx_bytes + G * C * d * el + T * E * 4, 0.0),
        "combine": (A * d * el + 3 * idx_bytes + T * N * d * el, 0.0),
        "tc_fc1_gelu": (A * d * el + w + 2 * A * f * el, gemm_flops),
        "tc_fc2": (A * f * el + w + A * d * el, gemm_flops),
        "tc_da_dgelu": (A * d * el + w + 2 * A * f * el, gemm_flops),
        "tc_dx": (A * f * el + w + A * d * el, gemm_flops),
        "tc_dw1": (A * (d + f) * el + G * d * f * el, gemm_flops),
        "tc_dw2": (A * (d + f) * el + G * d * f * el, gemm_flops),
        # router backward (outside the a1..a12 step; timed on its own).  router_grad:
        # dY and the kept Ye rows in, dgate and dlogits out, dX read and written,
        # W_r once per task (logits too without renormalisation).  router_dw: x and
        # dlogits in, dW_r and dbias out.
        "router_grad": (3 * T * N * d * el + A * d * el + 4 * idx_bytes + T * N * E * 4
                        + T * d * E * 4 + (T * N * E * 4 if cfg.flags & 2 else 0),
                        2.0 * A * d + 2.0 * T * N * k * d),
        "router_dw": (T * N * d * el + T * N * E * 4 + T * d * E * 4 + T * E * 4,
                      2.0 * T * N * d * E),
    }


def traffic_record(kernel, workload, path=None):
    """DRAM bytes per launch of `kernel` from the committed ncu summary
    (profiles/dram_traffic.json), if it was captured on `workload` and the
    kernel's source files still hash to the value recorded with the counters;
    else None."""
    import hashlib
    path = path or os.path.join(ROOT, "profiles", "dram_traffic.json")
    try:
        with open(path) as fh:
            data = json.load(fh)
        if data.get("workload") != workload:
            return None
        rec = data["kernels"][kernel]
        h = hashlib.sha256()
        for f in rec["source_files"]:
            with open(os.path.join(ROOT, f), "rb") as fh:
                h.update(fh.read())
        if h.hexdigest() != rec["sources_sha256"]:
            return None
        return float(rec["dram_bytes_per_launch_full_size"])
    except Exception:
        return None


# ----------------------------------------------------------------------------- multi-rank host logic
def max_over_ranks(values, dist=None, device="cpu"):
    """Element-wise max of a list of floats over all ranks of the default process
    group (identity without one).  The job is as slow as its slowest rank."""
    import torch
    t = torch.tensor([float(v) for v in values], dtype=torch.float64, device=device)
    if dist is not None and dist.is_available() and dist.is_initialized():
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(v) for v in t.tolist()]


def job_tokens_per_s(tokens_per_rank_step, world, ms_per_step):
    """Whole-job throughput under weak scaling: every rank runs its own full
    workload, so the job moves world x tokens_per_rank_step tokens per step."""
    return tokens_per_rank_step * world / (ms_per_step / 1e3)


def rank_weight_seed(rank):
    """Each rank draws its own experts (independent tasks per rank)."""
    return 1234 + rank


# ----------------------------------------------------------------------------- clocks
class ClockSampler:
    """nvidia-smi clock / throttle sampling while the timed region runs."""

    QUERY = ("index,uuid,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, uuid):
        self.uuid = uuid
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "--query-gpu=" + self.QUERY, "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except Exception:
            self.proc.kill()
            out, _ = self.proc.communicate()
        rows = []
        for line in out.splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 10:
                continue
            if self.uuid and self.uuid not in parts[1]:
                continue
            rows.append(parts)
        if not rows:
            return None
        def num(s):
            try:
                return float(s)
            except ValueError:
                return float("nan")
        sm = [num(r[2]) for r in rows]
        mx = max(num(r[3]) for r in rows)
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[6 + i] == "Active"})
        loaded = [v for v in sm if v > 0.5 * mx] or sm
        return {"sm_mhz": statistics.median(loaded), "sm_max_mhz": mx, "reasons": reasons,
                "samples": len(rows), "power_w_max": max(num(r[4]) for r in rows)}


# ----------------------------------------------------------------------------- ours
def run_ours(args, cfg, rank, world, local_rank):
    import torch
    import paper_2608_16188_gb300 as vm

    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)

    p = vm.problem(cfg.T, cfg.N, cfg.d, cfg.f, cfg.E, cfg.k, cfg.cf, cfg.dtype, cfg.flags)
    C = vm.vmoe_problem_capacity(p)
    cfg = cfg.with_(capacity=C)
    # Tokens, routers and dY follow the seeded recipe; the 5.1 GB of expert weights
    # are drawn on the device with the same distribution (rank-dependent seed).
    inp = workloads.make_inputs(cfg, with_weights=False)
    inp = {k2: (None if v is None else v.to(dev)) for k2, v in inp.items()}
    inp["w1"], inp["w2"] = workloads.make_weights_fast(cfg, dev, seed=rank_weight_seed(rank))
    runner = vm.StepRunner(p, inp)
    stream = torch.cuda.current_stream(dev)

    def barrier():
        if dist is not None:
            dist.barrier()

    for _ in range(args.warmup):
        runner.step(stream)
    torch.cuda.synchronize(dev)
    st = vm.vmoe_device_status()
    if st != 0:
        raise RuntimeError("device status after warm-up: " + vm.status_string(st))
    loads = runner.b.load.flatten().tolist()

    # ---- device-timed region (inputs resident in HBM).  The kernel trace records
    # CUDA events between launches, which would break the programmatic
    # dependent-launch chain of a step, so per-kernel times come from a separate
    # traced pass after it.
    props = torch.cuda.get_device_properties(dev)
    sampler = ClockSampler(str(getattr(props, "uuid", "")) or None)
    sampler.start()
    time.sleep(0.3)
    barrier()
    torch.cuda.synchronize(dev)
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        runner.step(stream)
    e1.record(stream)
    torch.cuda.synchronize(dev)
    barrier()
    clocks = sampler.stop()
    ms_total = e0.elapsed_time(e1)
    trace_steps = max(3, min(args.steps, 50))
    vm.vmoe_trace_enable(trace_steps * 32 + 64)
    for _ in range(trace_steps):
        runner.step(stream)
    torch.cuda.synchronize(dev)
    n_rec = vm.vmoe_trace_disable()
    per_kernel = {}
    for i in range(n_rec):
        name, ms = vm.vmoe_trace_get(i)
        per_kernel.setdefault(name, []).append(ms)
    step_launches = n_rec // trace_steps

    # ---- end-to-end region: every step uploads its x and dY from pinned host
    # memory and reads y and dX back into pinned host memory.  HostPipeline
    # overlaps those copies with compute (a copy stream, two buffer slots); the
    # same loop with the copies in line on the compute stream is reported beside it.
    x_h = inp["x"].cpu().pin_memory()
    dy_h = inp["dy"].cpu().pin_memory()
    outs = [(torch.empty(runner.b.y.shape, dtype=runner.b.y.dtype).pin_memory(),
             torch.empty(runner.b.dx.shape, dtype=runner.b.dx.dtype).pin_memory())
            for _ in range(2)]
    e2e_steps = max(1, min(args.steps, 50))
    weights = {k2: v for k2, v in inp.items() if k2 not in ("x", "dy")}
    pipe = vm.HostPipeline(p, weights, runner.b, dev)

    def e2e_pipelined(n):
        pipe.run([(x_h, dy_h)] * n, [outs[i % 2] for i in range(n)], stream)
        torch.cuda.synchronize(dev)

    def e2e_serial(n):
        for i in range(n):
            inp["x"].copy_(x_h, non_blocking=True)
            inp["dy"].copy_(dy_h, non_blocking=True)
            runner.step(stream)
            outs[i % 2][0].copy_(runner.b.y, non_blocking=True)
            outs[i % 2][1].copy_(runner.b.dx, non_blocking=True)
        torch.cuda.synchronize(dev)

    e2e_times = {}
    for name, fn in (("pipelined", e2e_pipelined), ("serial", e2e_serial)):
        fn(2)
        barrier()
        torch.cuda.synchronize(dev)
        t0 = time.perf_counter()
        fn(e2e_steps)
        e2e_times[name] = time.perf_counter() - t0
        barrier()
    e2e_s, e2e_serial_s = e2e_times["pipelined"], e2e_times["serial"]
    x_h0, dy_h0 = x_h, dy_h
    y_h, dx_h = outs[0]
    st = vm.vmoe_device_status()
    if st != 0:
        raise RuntimeError("device status after timing: " + vm.status_string(st))

    # ---- router backward on its own (the gating network's gradient), L2 flushed
    # between iterations -- a 256 MiB write, then a 256 MiB read so that the
    # lines left in L2 are clean and the next call pays no write-back for them;
    # the trace times each of its kernels
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    flush_r = torch.ones(64 << 20, dtype=torch.float32, device=dev)
    rb_steps = max(3, min(args.steps, 100))
    for _ in range(3):
        runner.router_backward(stream)
    vm.vmoe_trace_enable(rb_steps * 3 + 16)
    for _ in range(rb_steps):
        flush.zero_()
        flush_r.sum()
        runner.router_backward(stream)
    torch.cuda.synchronize(dev)
    rb_rec = vm.vmoe_trace_disable()
    rb_kernel = {}
    for i in range(rb_rec):
        name, ms = vm.vmoe_trace_get(i)
        rb_kernel.setdefault(name, []).append(ms)
    del flush, flush_r
    st = vm.vmoe_device_status()
    if st != 0:
        raise RuntimeError("device status after router backward: " + vm.status_string(st))

    # ---- the expert backward under a 64 MiB dH budget (the static-scratch entry
    # point, which plans slices with the cross-task DP and synchronises once to
    # read the loads), against the same backward with a full workspace
    b = runner.b
    bw_args = (p, b.xe, b.h, b.a, inp["w1"], inp["w2"], b.dye, b.load, b.dxe, b.dw1, b.dw2)
    for _ in range(2):
        vm.vmoe_expert_bwd_static_scratch(*bw_args)
    torch.cuda.synchronize(dev)
    bw_calls = 10
    vm.vmoe_trace_enable(bw_calls * 40 + 16)
    t0 = time.perf_counter()
    for _ in range(bw_calls):
        vm.vmoe_expert_bwd_static_scratch(*bw_args)
    torch.cuda.synchronize(dev)
    bw_wall = (time.perf_counter() - t0) / bw_calls
    n_bw = vm.vmoe_trace_disable()
    bw_kernel_ms = sum(vm.vmoe_trace_get(i)[1] for i in range(n_bw)) / bw_calls
    st = vm.vmoe_device_status()
    if st != 0:
        raise RuntimeError("device status after the budgeted backward: " + vm.status_string(st))

    # ---- max over ranks
    ms_total, e2e_s, e2e_serial_s = max_over_ranks([ms_total, e2e_s, e2e_serial_s], dist, dev)
    tokens_per_step = cfg.T * cfg.N * world
    ms_step = ms_total / args.steps
    value = job_tokens_per_s(cfg.T * cfg.N, world, ms_step)

    counts = model_counts(cfg, loads)
    peaks = load_peaks()
    kstats = {}
    # the committed DRAM records hold for their workload at its full task count only
    # (a --tasks prefix keeps the name but not the sizes)
    traffic_key = cfg.name if cfg.T == workloads.CONFIGS[cfg.name].T else None
    for name, ms_list in per_kernel.items():
        avg = sum(ms_list) / len(ms_list)
        by, fl = counts.get(name, (0, 0.0))
        launches_per_step = len(ms_list) / trace_steps
        tr = traffic_record(name, traffic_key)
        kstats[name] = {"launches": len(ms_list), "ms_avg": round(avg, 5),
                        "share": 0.0,
                        "gb_s": round(by / (avg * 1e-3) / 1e9, 1) if by else None,
                        # on the measured DRAM traffic (the committed ncu launch list)
                        "dram_gb_s": round(tr / (avg * 1e-3) / 1e9, 1) if tr else None,
                        "tflop_s": round(fl / (avg * 1e-3) / 1e12, 2) if fl else None,
                        "launches_per_step": launches_per_step}
    busy = sum(v["ms_avg"] * v["launches"] for v in kstats.values())
    for v in kstats.values():
        v["share"] = round(v["ms_avg"] * v["launches"] / busy, 4) if busy else 0.0
    dom = max(kstats, key=lambda n: kstats[n]["ms_avg"] * kstats[n]["launches"])
    dom_bytes, dom_flops = counts.get(dom, (0, 0.0))
    dom_ms = kstats[dom]["ms_avg"]
    achieved = dom_bytes / (dom_ms * 1e-3) / 1e9
    roofline = {"kernel": dom, "bound": "hbm", "achieved": round(achieved, 1),
                "peak": peaks["hbm_gbs"], "unit": "GB/s",
                "frac": round(achieved / peaks["hbm_gbs"], 4),
                "traffic": traffic_record(dom, traffic_key),
                "algorithmic_bytes_per_launch": dom_bytes,
                "peak_source": peaks["source"] + " (MEASURED_PEAKS.json hbm_gbs)"}
    rb_stats = {}
    for name, ms_list in rb_kernel.items():
        avg = sum(ms_list) / len(ms_list)
        by, fl = counts.get(name, (0, 0.0))
        rb_stats[name] = {"launches": len(ms_list), "ms_avg": round(avg, 5),
                          "gb_s": round(by / (avg * 1e-3) / 1e9, 1) if by else None,
                          "algorithmic_bytes_per_launch": by}
    rb_ms = sum(v["ms_avg"] for v in rb_stats.values())
    rb_dom = max(rb_stats, key=lambda n: rb_stats[n]["ms_avg"]) if rb_stats else None
    router_bwd = None
    if rb_dom is not None:
        rb_ach = rb_stats[rb_dom]["gb_s"] or 0.0
        router_bwd = {
            "what": "vmoe_router_bwd: dgate, dlogits, dW_r, dbias, dX += dlogits W_r^T "
                    "(gating-network gradient; not part of the a1..a12 step above)",
            "ms_per_call": round(rb_ms, 5), "calls": rb_steps,
            "l2": "flushed before every call (256 MiB write, then 256 MiB read: clean lines)",
            "kernels": rb_stats,
            "roofline": {"kernel": rb_dom, "bound": "hbm", "achieved": rb_ach,
                         "peak": peaks["hbm_gbs"], "unit": "GB/s",
                         "frac": round(rb_ach / peaks["hbm_gbs"], 4),
                         "traffic": traffic_record(rb_dom, traffic_key),
                         "peak_source": peaks["source"] + " (MEASURED_PEAKS.json hbm_gbs)"},
            "step_with_router_bwd_tokens_per_s": round(
                job_tokens_per_s(cfg.T * cfg.N, world, ms_step + rb_ms), 1),
        }
    gemm_flops = sum(counts[n][1] * kstats[n]["launches_per_step"] for n in kstats if n.startswith("tc_"))
    tflops = gemm_flops / (ms_step * 1e-3) / 1e12 * world
    h2d = (x_h0.numel() * x_h0.element_size() + dy_h0.numel() * dy_h0.element_size())
    d2h = (y_h.numel() * y_h.element_size() + dx_h.numel() * dx_h.element_size())
    out = {
        "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_step, 5),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded; expert weights drawn on device)",
        "config": {"workload": cfg.name + ": " + cfg.note, "T": cfg.T, "tokens_per_task": cfg.N,
                   "images_per_task": cfg.images_per_task, "d_model": cfg.d, "d_ff": cfg.f,
                   "E": cfg.E, "k": cfg.k, "capacity_factor": cfg.cf, "capacity": C,
                   "kept_assignments": int(sum(loads)),
                   "tasks_total": cfg.T * world, "l2": L2_NOTE},
        "tflops": round(tflops, 2),
        "bf16_peak_frac": round(tflops / world / peaks["bf16_tflops_sustained"], 4),
        "bf16_peak_note": "grouped-GEMM flops on kept rows / step time, vs measured sustained bf16 peak",
        "roofline": roofline,
        "kernels": kstats,
        "gpu_launches": int(step_launches * args.steps),
        "launch": "programmatic dependent launch " + ("off (VMOE_PDL=0)" if os.environ.get("VMOE_PDL") == "0" else "on"),
        "e2e": {"value": round(tokens_per_step * e2e_steps / e2e_s, 1), "unit": UNIT,
                "h2d_bytes_per_step": h2d * world, "d2h_bytes_per_step": d2h * world,
                "steps": e2e_steps,
                "how": "HostPipeline: per step x, dY up from pinned host memory and y, dX back, "
                       "on a copy stream overlapped with compute (two buffer slots)",
                "serial_value": round(tokens_per_step * e2e_steps / e2e_serial_s, 1)},
        "clocks": clocks,
        "router_bwd": router_bwd,
        "budgeted_bwd": {
            "what": "vmoe_expert_bwd_static_scratch: the expert backward with dH limited to the "
                    "library's 64 MiB array, groups in slices planned by the cross-task DP",
            "budget_bytes": vm.VMOE_STATIC_SCRATCH_BYTES,
            "full_workspace_bytes": vm.vmoe_expert_bwd_workspace_size(p),
            "ms_per_call_wall": round(bw_wall * 1e3, 4),
            "kernel_ms_per_call": round(bw_kernel_ms, 4),
            "launches_per_call": n_bw // bw_calls,
            "full_workspace_kernel_ms": round(sum(kstats[k]["ms_avg"] for k in
                                                  ("tc_da_dgelu", "tc_dx", "tc_dw1", "tc_dw2")
                                                  if k in kstats), 4),
        },
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        out["cpu_baseline"] = cpu_baseline(cfg, budget_s=args.cpu_budget)
    if dist is not None:
        dist.barrier()
        dist.destroy_process_group()
    return out


# ----------------------------------------------------------------------------- oracle legs
_TASK0 = {}


def _task0_inputs(cfg):
    if cfg.name not in _TASK0:
        _TASK0[cfg.name] = workloads.make_inputs(cfg, tasks=[0])
    return _TASK0[cfg.name]


def _oracle_tokens_per_s(cfg, n_tokens, repeats=1):
    """Wall time of the fp64 oracle on one task of `cfg` cut to its first
    n_tokens tokens (capacity recomputed for that N)."""
    import oracle
    sub = cfg.with_(T=1, N=n_tokens, capacity=0)
    inp = _task0_inputs(cfg)
    x = inp["x"][:, :n_tokens]
    dy = inp["dy"][:, :n_tokens]
    C = oracle.capacity(n_tokens, sub.E, sub.k, sub.cf)
    t0 = time.perf_counter()
    for _ in range(repeats):
        oracle.step(x, inp["w_router"], inp["bias"], inp["w1"], inp["w2"], dy, sub.k, C, sub.flags)
    dt = (time.perf_counter() - t0) / repeats
    return n_tokens / dt, dt


def cpu_baseline(cfg, budget_s=20.0):
    """The oracle on a bounded sample of the workload: whole tasks (1576 tokens each
    at T17) when one task fits the budget, else task 0 cut to fewer tokens."""
    import oracle
    probe_tokens = 64
    _, dt = _oracle_tokens_per_s(cfg, probe_tokens)
    n = int(max(probe_tokens, min(cfg.N, probe_tokens * budget_s / max(dt, 1e-3))))
    if n < cfg.N:
        v, dt = _oracle_tokens_per_s(cfg, n)
        sample = "one fp64 step of task 0 cut to its first %d of %d tokens" % (n, cfg.N)
    else:
        _, dt1 = _oracle_tokens_per_s(cfg, cfg.N)
        tasks = int(max(1, min(cfg.T, budget_s / max(dt1, 1e-3))))
        inp = workloads.make_inputs(cfg, tasks=range(tasks))
        C = oracle.capacity(cfg.N, cfg.E, cfg.k, cfg.cf)
        t0 = time.perf_counter()
        oracle.step(inp["x"], inp["w_router"], inp["bias"], inp["w1"], inp["w2"], inp["dy"],
                    cfg.k, C, cfg.flags)
        dt = time.perf_counter() - t0
        v = tasks * cfg.N / dt
        sample = "one fp64 step of the first %d of %d tasks (%d tokens)" % (tasks, cfg.T,
                                                                           tasks * cfg.N)
    return {"value": round(v, 2), "unit": UNIT, "cores": oracle.num_threads(), "kind": "oracle",
            "sample": sample + ", %.1f s on host cores" % dt}


def run_reference(args, cfg):
    import oracle
    probe = 32
    _, dt = _oracle_tokens_per_s(cfg, probe)
    per_step_budget = max(1.0, 150.0 / max(1, args.steps + args.warmup))
    n = int(max(16, min(cfg.N, probe * per_step_budget / max(dt, 1e-3))))
    for _ in range(args.warmup):
        _oracle_tokens_per_s(cfg, n)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        _oracle_tokens_per_s(cfg, n)
    el = time.perf_counter() - t0
    value = n * args.steps / el
    sample = ("fp64 oracle step on task 0 of %s cut to its first %d of %d tokens per step "
              "(capacity recomputed for that token count)" % (cfg.name, n, cfg.N))
    return {"impl": "reference", "metric": METRIC, "value": round(value, 3), "unit": UNIT,
            "n_gpus": 1, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(el / args.steps * 1e3, 3), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded)",
            "config": {"workload": cfg.name + ": " + cfg.note, "T": cfg.T, "tokens_per_task": cfg.N,
                       "d_model": cfg.d, "d_ff": cfg.f, "E": cfg.E, "k": cfg.k,
                       "capacity_factor": cfg.cf},
            "cpu_baseline": {"value": round(value, 3), "unit": UNIT, "cores": oracle.num_threads(),
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": round(value, 3), "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=300)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--config", default=workloads.HEADLINE, choices=list(workloads.CONFIGS))
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-budget", type=float, default=20.0,
                    help="seconds of oracle work for the cpu_baseline sample")
    ap.add_argument("--tasks", type=int, default=0,
                    help="run only the first TASKS tasks of the workload (same per-group shapes; "
                         "used to size profiler captures)")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if world != args.gpus and "RANK" in os.environ:
        ap.error("--gpus %d but WORLD_SIZE=%d" % (args.gpus, world))
    cfg = workloads.CONFIGS[args.config]
    if args.tasks:
        cfg = cfg.with_(T=min(args.tasks, cfg.T))
    if args.impl == "reference":
        if rank != 0:
            return
        print(json.dumps(run_reference(args, cfg)), flush=True)
        return
    out = run_ours(args, cfg, rank, world, local_rank)
    if rank == 0:
        print(json.dumps(out), flush=True)


if __name__ == "__main__":
    main()
