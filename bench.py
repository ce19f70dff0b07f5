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
L2_BYTES = 129e6          # GB300 L2
FLUSH_BELOW = 16 * L2_BYTES  # flush L2 between timed steps when the weights are smaller
# the other workloads timed by the default run (parity cases, reported under "workloads")
SECONDARY = ("vits_t4", "vitb_t6", "skew_t8", "tiny_fp32")


def weight_bytes(cfg):
    el = 2 if cfg.dtype == "bf16" else 4
    return 2 * cfg.T * cfg.E * cfg.d * cfg.f * el


def l2_policy(cfg):
    """(flush, note): whether L2 is flushed between timed steps, and why."""
    wb = weight_bytes(cfg)
    if wb < FLUSH_BELOW:
        return True, ("L2 flushed before every timed step (256 MiB written, then 256 MiB read): "
                      "the %.2f GB of expert weights are %.1fx the 129 MB L2" % (wb / 1e9, wb / L2_BYTES))
    return False, ("inputs larger than L2: every step streams %.2f GB of expert weights "
                   "(plus as many bytes of weight gradients), %.0fx the 129 MB L2" % (wb / 1e9, wb / L2_BYTES))


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


def traffic_record(kernel, workload, algo_bytes, path=None):
    """DRAM bytes per launch of `kernel` at the full workload, from the committed
    ncu record (profiles/dram_traffic.json), or None.

    The record holds, per workload, one-kernel captures on a prefix of its tasks
    (a few GB on the device): the launch's dram__bytes_read.sum +
    dram__bytes_write.sum and its algorithmic bytes.  Tasks are independent and
    their groups drawn from the same distribution, so a kernel's traffic grows
    with the work it is given: the full-size figure is the measured one times
    algo_bytes (the full launch's algorithmic bytes) over the prefix's.  None
    when there is no record for the workload or kernel, or when the kernel's
    source files no longer hash to the value recorded with the counters.
    """
    import hashlib
    path = path or os.path.join(ROOT, "profiles", "dram_traffic.json")
    try:
        with open(path) as fh:
            data = json.load(fh)
        rec = data["workloads"][workload]["kernels"][kernel]
        h = hashlib.sha256()
        for f in rec["source_files"]:
            with open(os.path.join(ROOT, f), "rb") as fh:
                h.update(fh.read())
        if h.hexdigest() != rec["sources_sha256"]:
            return None
        return float(rec["dram_bytes_per_launch"]) * float(algo_bytes) / float(rec["algorithmic_bytes_per_launch"])
    except Exception:
        return None


# Source files behind each kernel name of the trace (for the traffic record's hash).
KERNEL_SOURCES = {
    "route_topk": ["route.cu", "route_tc.cu", "topk.cuh", "gemm_tc.cuh", "common.cuh"],
    "capacity_scan": ["route.cu", "common.cuh"],
    "dispatch": ["permute.cu", "common.cuh"],
    "combine": ["permute.cu", "common.cuh"],
    "tc_fc1_gelu": ["gemm_tc.cuh", "gemm_tc2.cuh", "gemm_tc_fwd.cu", "common.cuh"],
    "tc_fc2": ["gemm_tc.cuh", "gemm_tc2.cuh", "gemm_tc_fwd.cu", "common.cuh"],
    "tc_da_dgelu": ["gemm_tc.cuh", "gemm_tc2.cuh", "gemm_tc_bwd.cu", "common.cuh"],
    "tc_dx": ["gemm_tc.cuh", "gemm_tc2.cuh", "gemm_tc_bwd.cu", "common.cuh"],
    "tc_dw1": ["gemm_tc.cuh", "gemm_tc2.cuh", "gemm_tc_bwd.cu", "common.cuh"],
    "tc_dw2": ["gemm_tc.cuh", "gemm_tc2.cuh", "gemm_tc_bwd.cu", "common.cuh"],
    "router_grad": ["router_bwd.cu", "common.cuh"],
    "router_dw": ["router_bwd.cu", "router_dw_tc.cu", "common.cuh"],
}
# Kernel-name patterns (ncu -k regex) of the library's kernels, per trace name.
KERNEL_REGEX = {
    "route_topk": "route_", "capacity_scan": "capacity_scan", "dispatch": "dispatch_kernel",
    "combine": "combine_kernel", "router_grad": "router_grad", "router_dw": "router_dw",
}


def sources_sha256(kernel):
    import hashlib
    h = hashlib.sha256()
    for f in KERNEL_SOURCES[kernel]:
        with open(os.path.join(ROOT, "paper_2608_16188_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()


def write_traffic_record(workload, tasks, plain_json, captures, path=None):
    """Writes profiles/dram_traffic.json's entry for `workload` from ncu captures.

    plain_json: bench.py's JSON line of the same prefix run without ncu (it gives
    each kernel's algorithmic bytes per launch at that prefix); captures: pairs
    (trace kernel name, ncu --csv log of `--metrics dram__bytes_read.sum,
    dram__bytes_write.sum -k regex:<kernel> -c 1` on that run).
    """
    import csv
    path = path or os.path.join(ROOT, "profiles", "dram_traffic.json")
    with open(plain_json) as fh:
        plain = json.loads(fh.read().strip().splitlines()[-1])
    algo = {k: v.get("algorithmic_bytes_per_launch") for k, v in plain["kernels"].items()}
    algo.update({k: v.get("algorithmic_bytes_per_launch")
                 for k, v in ((plain.get("router_bwd") or {}).get("kernels") or {}).items()})
    try:
        with open(path) as fh:
            data = json.load(fh)
    except Exception:
        data = {}
    data["about"] = ("DRAM bytes (dram__bytes_read.sum + dram__bytes_write.sum) of one launch of each "
                     "library kernel, captured by ncu on a prefix of the workload's tasks (one kernel, "
                     "one launch, a few GB on the device), with that launch's algorithmic bytes; "
                     "bench.py scales them to the full workload by the algorithmic bytes and drops a "
                     "record once the kernel's sources change (sources_sha256).")
    wl = data.setdefault("workloads", {}).setdefault(workload, {})
    wl.pop("tasks", None)  # per kernel: captured_at_tasks
    kern = wl.setdefault("kernels", {})
    for name, log in captures:
        vals = {}
        with open(log) as fh:
            lines = [ln for ln in fh if ln.startswith('"')]
        for row in csv.DictReader(lines):
            if row.get("Metric Name") in ("dram__bytes_read.sum", "dram__bytes_write.sum"):
                unit = row.get("Metric Unit", "byte")
                scale = {"byte": 1, "Kbyte": 1e3, "Mbyte": 1e6, "Gbyte": 1e9}.get(unit, 1)
                vals[row["Metric Name"]] = float(row["Metric Value"].replace(",", "")) * scale
        if len(vals) != 2 or not algo.get(name):
            continue
        kern[name] = {"dram_bytes_per_launch": int(sum(vals.values())),
                      "algorithmic_bytes_per_launch": int(algo[name]),
                      "captured_at_tasks": tasks,
                      "source_files": ["paper_2608_16188_gb300/csrc/" + f for f in KERNEL_SOURCES[name]],
                      "sources_sha256": sources_sha256(name)}
    with open(path, "w") as fh:
        json.dump(data, fh, indent=1, sort_keys=True)
        fh.write("\n")


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
def l2_flusher(dev):
    """Evicts L2: a 256 MiB write, then a 256 MiB read so that the lines left in
    L2 are clean and the next step pays no write-back for them."""
    import torch
    wbuf = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    rbuf = torch.ones(64 << 20, dtype=torch.float32, device=dev)

    def flush():
        wbuf.zero_()
        rbuf.sum()
    return flush


def time_steps(step, stream, steps, flush=None):
    """Device time (ms) of `steps` calls of step(stream): one event pair around
    the whole loop, or -- with `flush` -- one pair per step with L2 flushed before
    each (the flush outside the timed pairs)."""
    import torch
    if flush is None:
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(steps):
            step(stream)
        e1.record(stream)
        e1.synchronize()
        return e0.elapsed_time(e1)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(steps)]
    for a, b in ev:
        flush()
        a.record(stream)
        step(stream)
        b.record(stream)
    ev[-1][1].synchronize()
    return sum(a.elapsed_time(b) for a, b in ev)


def traced_kernels(vm, step, stream, steps, flush=None):
    """Per-kernel device times from the library's event trace over `steps` more
    steps (L2 flushed before each with `flush`): {name: [ms, ...]}, launches/step."""
    import torch
    vm.vmoe_trace_enable(steps * 32 + 64)
    for _ in range(steps):
        if flush is not None:
            flush()
        step(stream)
    torch.cuda.synchronize()
    n_rec = vm.vmoe_trace_disable()
    per_kernel = {}
    for i in range(n_rec):
        name, ms = vm.vmoe_trace_get(i)
        per_kernel.setdefault(name, []).append(ms)
    return per_kernel, n_rec // steps


def kernel_stats(per_kernel, trace_steps, counts, traffic_key=None):
    """Per-kernel launches, mean time, share of the step's kernel time, GB/s on
    algorithmic bytes (and on the measured DRAM traffic where a record exists)."""
    kstats = {}
    for name, ms_list in per_kernel.items():
        avg = sum(ms_list) / len(ms_list)
        by, fl = counts.get(name, (0, 0.0))
        tr = traffic_record(name, traffic_key, by) if (traffic_key and by) else None
        kstats[name] = {"launches": len(ms_list), "ms_avg": round(avg, 5), "share": 0.0,
                        "gb_s": round(by / (avg * 1e-3) / 1e9, 1) if by else None,
                        "dram_gb_s": round(tr / (avg * 1e-3) / 1e9, 1) if tr else None,
                        "tflop_s": round(fl / (avg * 1e-3) / 1e12, 2) if fl else None,
                        "algorithmic_bytes_per_launch": by,
                        "launches_per_step": len(ms_list) / trace_steps}
    busy = sum(v["ms_avg"] * v["launches"] for v in kstats.values())
    for v in kstats.values():
        v["share"] = round(v["ms_avg"] * v["launches"] / busy, 4) if busy else 0.0
    return kstats


def roofline_of(kstats, counts, peaks, traffic_key=None):
    """Roofline line of the dominant kernel (largest share of the step)."""
    dom = max(kstats, key=lambda n: kstats[n]["ms_avg"] * kstats[n]["launches"])
    dom_bytes, _ = counts.get(dom, (0, 0.0))
    achieved = dom_bytes / (kstats[dom]["ms_avg"] * 1e-3) / 1e9
    return {"kernel": dom, "bound": "hbm", "achieved": round(achieved, 1),
            "peak": peaks["hbm_gbs"], "unit": "GB/s", "frac": round(achieved / peaks["hbm_gbs"], 4),
            "traffic": traffic_record(dom, traffic_key, dom_bytes) if traffic_key else None,
            "algorithmic_bytes_per_launch": dom_bytes,
            "peak_source": peaks["source"] + " (MEASURED_PEAKS.json hbm_gbs)"}


def combined_roofline(kstats, counts, peaks, ms_step, dtype):
    """Fraction of the step's combined roofline: sum over its launches of
    max(algorithmic bytes / HBM peak, flops / tensor peak), over the step time.
    bf16 contractions take the measured sustained bf16 peak; fp32 ones (CUDA
    cores) are counted on bytes alone."""
    t = 0.0
    for name, v in kstats.items():
        by, fl = counts.get(name, (0, 0.0))
        t_b = by / (peaks["hbm_gbs"] * 1e9)
        t_f = fl / (peaks["bf16_tflops_sustained"] * 1e12) if dtype == "bf16" else 0.0
        t += v["launches_per_step"] * max(t_b, t_f)
    return {"t_roof_ms": round(t * 1e3, 4), "frac": round(t * 1e3 / ms_step, 4) if ms_step else None}


def measure_secondary(vm, cfg, dev, stream, steps, warmup, peaks, seed):
    """One other workload (a parity case of the same method): device-timed step,
    per-kernel times, its dominant kernel's roofline and its combined-roofline
    fraction.  Inputs resident in HBM; L2 flushed between steps where the
    weights are small enough for L2 to matter."""
    import torch
    p = vm.problem(cfg.T, cfg.N, cfg.d, cfg.f, cfg.E, cfg.k, cfg.cf, cfg.dtype, cfg.flags)
    C = vm.vmoe_problem_capacity(p)
    cfg = cfg.with_(capacity=C)
    inp = workloads.make_inputs(cfg, with_weights=False)
    inp = {k2: (None if v is None else v.to(dev)) for k2, v in inp.items()}
    inp["w1"], inp["w2"] = workloads.make_weights_fast(cfg, dev, seed=seed)
    runner = vm.StepRunner(p, inp)
    flush_on, note = l2_policy(cfg)
    flush = l2_flusher(dev) if flush_on else None
    for _ in range(warmup):
        runner.step(stream)
    torch.cuda.synchronize(dev)
    loads = runner.b.load.flatten().tolist()
    ms = time_steps(runner.step, stream, steps, flush) / steps
    per_kernel, _ = traced_kernels(vm, runner.step, stream, min(steps, 20), flush)
    st = vm.vmoe_device_status()
    if st != 0:
        raise RuntimeError("device status after %s: %s" % (cfg.name, vm.status_string(st)))
    counts = model_counts(cfg, loads)
    traffic_key = cfg.name
    kstats = kernel_stats(per_kernel, min(steps, 20), counts, traffic_key)
    gemm_flops = sum(counts[n][1] * kstats[n]["launches_per_step"] for n in kstats if n.startswith("tc_"))
    out = {"config": {"workload": cfg.name + ": " + cfg.note, "T": cfg.T, "tokens_per_task": cfg.N,
                      "d_model": cfg.d, "d_ff": cfg.f, "E": cfg.E, "k": cfg.k, "capacity_factor": cfg.cf,
                      "capacity": C, "kept_assignments": int(sum(loads)), "dtype": cfg.dtype, "l2": note},
           "value": round(cfg.T * cfg.N / (ms * 1e-3), 1), "unit": UNIT, "ms_per_step": round(ms, 5),
           "steps": steps, "tflops": round(gemm_flops / (ms * 1e-3) / 1e12, 2),
           "roofline": roofline_of(kstats, counts, peaks, traffic_key),
           "combined_roofline": combined_roofline(kstats, counts, peaks, ms, cfg.dtype),
           "kernels": kstats}
    del runner, inp
    torch.cuda.empty_cache()
    return out


def measure_attention(vm, cfg, heads, dev, stream, steps, warmup, peaks, seed):
    """The attention-expert variant of the step at cfg's shape: route, dispatch,
    vmoe_attn_expert_fwd, combine, weighted dispatch of dY, vmoe_attn_expert_bwd,
    combine of dX -- H-head attention (head dimension 64) among each group's
    routed tokens in place of the FFN experts.  Weights drawn on the device."""
    import torch
    p = vm.problem(cfg.T, cfg.N, cfg.d, cfg.f, cfg.E, cfg.k, cfg.cf, cfg.dtype, cfg.flags)
    C = vm.vmoe_problem_capacity(p)
    inp = workloads.make_inputs(cfg.with_(capacity=C), with_weights=False)
    inp = {k2: (None if v is None else v.to(dev)) for k2, v in inp.items()}
    hd = heads * 64
    g = torch.Generator(device=dev)
    g.manual_seed(seed)
    G, d = cfg.T * cfg.E, cfg.d
    wqkv = (torch.randn((G, d, 3 * hd), generator=g, device=dev) / d ** 0.5).to(torch.bfloat16)
    wo = (torch.randn((G, hd, d), generator=g, device=dev) / hd ** 0.5).to(torch.bfloat16)
    b = vm.Buffers(p)
    e = lambda *sh, dt=torch.bfloat16: torch.empty(sh, dtype=dt, device=dev)  # noqa: E731
    qkv, o, ye, lse = e(G, C, 3 * hd), e(G, C, hd), e(G, C, d), e(G, heads, C, dt=torch.float32)
    dxe, dwqkv, dwo = e(G, C, d), e(G, d, 3 * hd), e(G, hd, d)
    ws = torch.empty(vm.vmoe_attn_expert_bwd_workspace_size(p, heads), dtype=torch.uint8, device=dev)

    def step(st):
        vm.vmoe_route(p, inp["x"], inp["w_router"], inp["bias"], b.logits, b.idx, b.gate, b.slot, b.load, st)
        vm.vmoe_dispatch(p, inp["x"], None, b.idx, b.slot, b.load, b.xe, st)
        vm.vmoe_attn_expert_fwd(p, heads, b.xe, wqkv, wo, b.load, qkv, o, lse, ye, st)
        vm.vmoe_combine(p, ye, b.gate, b.idx, b.slot, b.y, st)
        vm.vmoe_dispatch(p, inp["dy"], b.gate, b.idx, b.slot, b.load, b.dye, st)
        vm.vmoe_attn_expert_bwd(p, heads, b.xe, qkv, o, lse, wqkv, wo, b.dye, b.load, dxe, dwqkv, dwo, ws,
                                stream=st)
        vm.vmoe_combine(p, dxe, None, b.idx, b.slot, b.dx, st)
    for _ in range(warmup):
        step(stream)
    torch.cuda.synchronize(dev)
    loads = b.load.flatten().tolist()
    ms = time_steps(step, stream, steps) / steps
    per_kernel, _ = traced_kernels(vm, step, stream, min(steps, 20))
    st = vm.vmoe_device_status()
    if st != 0:
        raise RuntimeError("device status after the attention experts: " + vm.status_string(st))
    A = int(sum(loads))
    sq = float(sum(L * L for L in loads))
    # flops on kept rows: projections 2 A d (3 hd + hd) forward, twice that backward;
    # the core 4 sum(L^2) hd forward (S and P V), 8 sum(L^2) hd backward (recomputed
    # S, dP, dQ, dK, dV minus the shared S)
    proj = 2.0 * A * d * 4 * hd
    core = 4.0 * sq * hd
    kst = {}
    for name, lst in per_kernel.items():
        kst[name] = {"launches": len(lst), "ms_avg": round(sum(lst) / len(lst), 5)}
    core_ms = sum(kst[n]["ms_avg"] for n in ("attn_fwd", "attn_bwd", "attn_bwd_dq", "attn_bwd_dkv") if n in kst)
    out = {"config": {"workload": cfg.name + " shape with attention experts (H=%d, head dim 64)" % heads,
                      "T": cfg.T, "tokens_per_task": cfg.N, "d_model": d, "E": cfg.E, "k": cfg.k,
                      "capacity": C, "heads": heads, "kept_assignments": A},
           "value": round(cfg.T * cfg.N / (ms * 1e-3), 1), "unit": UNIT, "ms_per_step": round(ms, 5),
           "steps": steps,
           "tflops": round((3 * proj + 3 * core) / (ms * 1e-3) / 1e12, 2),
           "core_ms_per_step": round(core_ms, 5),
           "core_tflop_s": round(3 * core / (core_ms * 1e-3) / 1e12, 2) if core_ms else None,
           "kernels": kst}
    del b, qkv, o, ye, dxe, dwqkv, dwo, ws, wqkv, wo
    torch.cuda.empty_cache()
    return out


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
    # Tokens, routers and dY follow the seeded recipe; the expert weights are drawn
    # on the device with the same distribution (rank-dependent seed).
    inp = workloads.make_inputs(cfg, with_weights=False)
    inp = {k2: (None if v is None else v.to(dev)) for k2, v in inp.items()}
    inp["w1"], inp["w2"] = workloads.make_weights_fast(cfg, dev, seed=rank_weight_seed(rank))
    runner = vm.StepRunner(p, inp)
    stream = torch.cuda.current_stream(dev)
    flush_on, l2_note = l2_policy(cfg)
    flush = l2_flusher(dev) if flush_on else None

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
    ms_total = time_steps(runner.step, stream, args.steps, flush)
    torch.cuda.synchronize(dev)
    barrier()
    clocks = sampler.stop()
    trace_steps = max(3, min(args.steps, 50))
    per_kernel, step_launches = traced_kernels(vm, runner.step, stream, trace_steps, flush)

    extras = not args.no_extras
    if extras:
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
        y_h, dx_h = outs[0]
        st = vm.vmoe_device_status()
        if st != 0:
            raise RuntimeError("device status after timing: " + vm.status_string(st))

        # ---- router backward on its own (the gating network's gradient), L2 flushed
        # between calls; the trace times each of its kernels
        rflush = flush or l2_flusher(dev)
        rb_steps = max(3, min(args.steps, 100))
        for _ in range(3):
            runner.router_backward(stream)
        vm.vmoe_trace_enable(rb_steps * 3 + 16)
        for _ in range(rb_steps):
            rflush()
            runner.router_backward(stream)
        torch.cuda.synchronize(dev)
        rb_rec = vm.vmoe_trace_disable()
        rb_kernel = {}
        for i in range(rb_rec):
            name, ms = vm.vmoe_trace_get(i)
            rb_kernel.setdefault(name, []).append(ms)
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
        # wall time per call without the kernel trace (its events between
        # launches would break the programmatic-dependent-launch chain) ...
        t0 = time.perf_counter()
        for _ in range(bw_calls):
            vm.vmoe_expert_bwd_static_scratch(*bw_args)
        torch.cuda.synchronize(dev)
        bw_wall = (time.perf_counter() - t0) / bw_calls
        # ... the full-workspace backward timed the same way, one call at a time
        full_args = bw_args + (b.workspace,)
        t0 = time.perf_counter()
        for _ in range(bw_calls):
            vm.vmoe_expert_bwd(*full_args)
            torch.cuda.synchronize(dev)
        full_wall = (time.perf_counter() - t0) / bw_calls
        # ... and the kernels' device times from a traced pass
        vm.vmoe_trace_enable(bw_calls * 64 + 16)
        for _ in range(bw_calls):
            vm.vmoe_expert_bwd_static_scratch(*bw_args)
        torch.cuda.synchronize(dev)
        n_bw = vm.vmoe_trace_disable()
        bw_kernel_ms = sum(vm.vmoe_trace_get(i)[1] for i in range(n_bw)) / bw_calls
        st = vm.vmoe_device_status()
        if st != 0:
            raise RuntimeError("device status after the budgeted backward: " + vm.status_string(st))
    else:
        e2e_s = e2e_serial_s = 0.0

    # ---- max over ranks
    ms_total, e2e_s, e2e_serial_s = max_over_ranks([ms_total, e2e_s, e2e_serial_s], dist, dev)
    tokens_per_step = cfg.T * cfg.N * world
    ms_step = ms_total / args.steps
    value = job_tokens_per_s(cfg.T * cfg.N, world, ms_step)

    counts = model_counts(cfg, loads)
    peaks = load_peaks()
    # DRAM records scale to the full task count only (a --tasks prefix keeps the
    # workload's name but not its sizes)
    traffic_key = cfg.name if cfg.T == workloads.CONFIGS[cfg.name].T else None
    kstats = kernel_stats(per_kernel, trace_steps, counts, traffic_key)
    roofline = roofline_of(kstats, counts, peaks, traffic_key)
    gemm_flops = sum(counts[n][1] * kstats[n]["launches_per_step"] for n in kstats if n.startswith("tc_"))
    tflops = gemm_flops / (ms_step * 1e-3) / 1e12 * world
    out = {
        "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_step, 5),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded; expert weights drawn on device)",
        "config": {"workload": cfg.name + ": " + cfg.note, "T": cfg.T, "tokens_per_task": cfg.N,
                   "images_per_task": cfg.images_per_task, "d_model": cfg.d, "d_ff": cfg.f,
                   "E": cfg.E, "k": cfg.k, "capacity_factor": cfg.cf, "capacity": C,
                   "kept_assignments": int(sum(loads)),
                   "tasks_total": cfg.T * world, "l2": l2_note},
        "tflops": round(tflops, 2),
        "bf16_peak_frac": round(tflops / world / peaks["bf16_tflops_sustained"], 4),
        "bf16_peak_note": "grouped-GEMM flops on kept rows / step time, vs measured sustained bf16 peak",
        "roofline": roofline,
        "combined_roofline": combined_roofline(kstats, counts, peaks, ms_step, cfg.dtype),
        "kernels": kstats,
        "gpu_launches": int(step_launches * args.steps),
        "launch": "programmatic dependent launch " + ("off (VMOE_PDL=0)" if os.environ.get("VMOE_PDL") == "0" else "on"),
        "clocks": clocks,
    }
    if extras:
        h2d = (x_h.numel() * x_h.element_size() + dy_h.numel() * dy_h.element_size())
        d2h = (y_h.numel() * y_h.element_size() + dx_h.numel() * dx_h.element_size())
        out["e2e"] = {"value": round(tokens_per_step * e2e_steps / e2e_s, 1), "unit": UNIT,
                      "h2d_bytes_per_step": h2d * world, "d2h_bytes_per_step": d2h * world,
                      "steps": e2e_steps,
                      "how": "HostPipeline: per step x, dY up from pinned host memory and y, dX back, "
                             "on a copy stream overlapped with compute (two buffer slots)",
                      "serial_value": round(tokens_per_step * e2e_steps / e2e_serial_s, 1)}
        rb_stats = {}
        for name, ms_list in rb_kernel.items():
            avg = sum(ms_list) / len(ms_list)
            by, fl = counts.get(name, (0, 0.0))
            rb_stats[name] = {"launches": len(ms_list), "ms_avg": round(avg, 5),
                              "gb_s": round(by / (avg * 1e-3) / 1e9, 1) if by else None,
                              "algorithmic_bytes_per_launch": by}
        rb_ms = sum(v["ms_avg"] for v in rb_stats.values())
        rb_dom = max(rb_stats, key=lambda n: rb_stats[n]["ms_avg"]) if rb_stats else None
        if rb_dom is not None:
            rb_ach = rb_stats[rb_dom]["gb_s"] or 0.0
            out["router_bwd"] = {
                "what": "vmoe_router_bwd: dgate, dlogits, dW_r, dbias, dX += dlogits W_r^T "
                        "(gating-network gradient; not part of the a1..a12 step above)",
                "ms_per_call": round(rb_ms, 5), "calls": rb_steps,
                "l2": "flushed before every call (256 MiB write, then 256 MiB read: clean lines)",
                "kernels": rb_stats,
                "roofline": {"kernel": rb_dom, "bound": "hbm", "achieved": rb_ach,
                             "peak": peaks["hbm_gbs"], "unit": "GB/s",
                             "frac": round(rb_ach / peaks["hbm_gbs"], 4),
                             "traffic": traffic_record(rb_dom, traffic_key,
                                                       rb_stats[rb_dom]["algorithmic_bytes_per_launch"])
                             if traffic_key else None,
                             "peak_source": peaks["source"] + " (MEASURED_PEAKS.json hbm_gbs)"},
                "step_with_router_bwd_tokens_per_s": round(
                    job_tokens_per_s(cfg.T * cfg.N, world, ms_step + rb_ms), 1),
            }
        out["budgeted_bwd"] = {
            "what": "vmoe_expert_bwd_static_scratch: the expert backward with dH limited to the "
                    "library's 64 MiB array, groups in slices planned by the cross-task DP",
            "budget_bytes": vm.VMOE_STATIC_SCRATCH_BYTES,
            "full_workspace_bytes": vm.vmoe_expert_bwd_workspace_size(p),
            "ms_per_call_wall": round(bw_wall * 1e3, 4),
            "full_workspace_ms_per_call_wall": round(full_wall * 1e3, 4),
            "kernel_ms_per_call": round(bw_kernel_ms, 4),
            "launches_per_call": n_bw // bw_calls,
            "full_workspace_kernel_ms": round(sum(kstats[k]["ms_avg"] for k in
                                                  ("tc_da_dgelu", "tc_dx", "tc_dw1", "tc_dw2")
                                                  if k in kstats), 4),
        }
    # ---- the other workloads (parity cases of the same method), rank 0 at N=1 only
    if rank == 0 and world == 1 and not args.headline_only:
        del runner
        torch.cuda.empty_cache()
        # a --tasks prefix (a profiling run) skips the other workloads and runs the
        # attention experts on the same prefix of the headline workload
        if not args.tasks:
            out["workloads"] = {name: measure_secondary(vm, workloads.CONFIGS[name], dev, stream,
                                                        args.aux_steps, args.warmup, peaks, seed=7)
                                for name in SECONDARY if name != cfg.name}
        att_cfg = workloads.CONFIGS[workloads.HEADLINE]
        if args.tasks:
            att_cfg = att_cfg.with_(T=min(args.tasks, att_cfg.T))
        out["attention_experts"] = measure_attention(vm, att_cfg, 12, dev, stream, args.aux_steps,
                                                     args.warmup, peaks, seed=9)
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
    ap.add_argument("--aux-steps", type=int, default=30,
                    help="timed steps of each other workload reported under 'workloads'")
    ap.add_argument("--headline-only", action="store_true",
                    help="time only --config (skip the other workloads)")
    ap.add_argument("--no-extras", action="store_true",
                    help="skip the end-to-end, router-backward and budgeted-backward legs")
    ap.add_argument("--write-traffic-record", nargs="+", metavar="ARG",
                    help="WORKLOAD TASKS PLAIN_JSON KERNEL=NCU_CSV ...: write profiles/dram_traffic.json "
                         "from one-kernel ncu captures of a --tasks prefix run, then exit")
    args = ap.parse_args()
    if args.write_traffic_record:
        wl, tasks, plain, *caps = args.write_traffic_record
        write_traffic_record(wl, int(tasks), plain, [tuple(c.split("=", 1)) for c in caps])
        return
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
