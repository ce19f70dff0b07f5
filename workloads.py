"""Seeded synthetic workloads shaped like the paper's multi-view V-MoE adaptation jobs.

This module holds the problem configurations and the seeded input generators.  It
contains none of the method's arithmetic and imports neither the oracle nor the
CUDA library, so it can feed both.

Recipe (the paper's CampReal / TrafficSim data are not available; these inputs
stand in for them, with the ViT shapes the paper uses: 197 tokens per image,
several images per task, one router and E experts per task):
  * every tensor gets its own ``torch.Generator`` seeded from
    (config index, task, tensor kind, expert) so that any single task or group
    can be regenerated alone;
  * x ~ N(0,1), W_r ~ N(0, 1/d), W1 ~ N(0, 1/d), W2 ~ N(0, 1/f), dY ~ N(0,1);
  * drifted tasks add a per-(task, expert) logit bias ~ N(0, 0.5^2);
  * the skewed-load case adds bias_e = -1.2 * ln(rank_e + 1) with rank a seeded
    per-task permutation of the experts (Zipf s = 1.2 popularity);
  * values are drawn in fp32 and rounded to bf16 for bf16 configurations
    (x, W1, W2, dY); W_r and the bias stay fp32.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field, replace

import torch

KIND_WR, KIND_BIAS, KIND_W1, KIND_W2, KIND_X, KIND_DY = range(6)


@dataclass(frozen=True)
class Config:
    name: str
    index: int
    T: int
    N: int
    d: int
    f: int
    E: int
    k: int
    cf: float
    dtype: str  # "f32" or "bf16"
    bias: str = "none"  # "none" | "drift" | "zipf"
    flags: int = 0
    capacity: int = 0
    images_per_task: int = 0
    note: str = field(default="", compare=False)

    @property
    def torch_dtype(self):
        return torch.float32 if self.dtype == "f32" else torch.bfloat16

    @property
    def G(self) -> int:
        return self.T * self.E

    def with_(self, **kw) -> "Config":
        return replace(self, **kw)


CONFIGS = {
    "tiny_fp32": Config("tiny_fp32", 0, T=2, N=64, d=64, f=256, E=4, k=2, cf=2.0, dtype="f32",
                        note="tiny V-MoE expert layer, fp32"),
    "vits_t4": Config("vits_t4", 1, T=4, N=8 * 197, d=384, f=1536, E=8, k=2, cf=1.25,
                      dtype="bf16", images_per_task=8, note="ViT-S-shaped layer, 4 tasks"),
    "vitb_t6": Config("vitb_t6", 2, T=6, N=16 * 197, d=768, f=3072, E=32, k=2, cf=1.25,
                      dtype="bf16", images_per_task=16, note="ViT-B-shaped layer, 6 tasks"),
    "vitb_t17": Config("vitb_t17", 3, T=17, N=8 * 197, d=768, f=3072, E=32, k=2, cf=1.25,
                       dtype="bf16", bias="drift", images_per_task=8,
                       note="ViT-B-shaped 17-task co-adaptation with drifted router logits"),
    "skew_t8": Config("skew_t8", 4, T=8, N=8 * 197, d=1024, f=4096, E=64, k=1, cf=1.0,
                      dtype="bf16", bias="zipf", images_per_task=8,
                      note="skewed expert load (Zipf 1.2), top-1, drops"),
}

# The 17-task ViT-B co-adaptation step is the headline workload.
HEADLINE = "vitb_t17"


def _seed(cfg_index: int, task: int, kind: int, expert: int = 0) -> int:
    return ((1000 * (cfg_index + 1) + task) * 16 + kind) * 8192 + expert


def _randn(shape, seed, std, device):
    g = torch.Generator(device="cpu")
    g.manual_seed(seed)
    out = torch.randn(shape, generator=g, dtype=torch.float32)
    if std != 1.0:
        out.mul_(std)
    return out.to(device) if device != "cpu" else out


def task_router(cfg: Config, t: int):
    """(W_r [d,E] fp32, bias [E] fp32 or None) of task t."""
    wr = _randn((cfg.d, cfg.E), _seed(cfg.index, t, KIND_WR), 1.0 / math.sqrt(cfg.d), "cpu")
    if cfg.bias == "drift":
        bias = _randn((cfg.E,), _seed(cfg.index, t, KIND_BIAS), 0.5, "cpu")
    elif cfg.bias == "zipf":
        g = torch.Generator(device="cpu")
        g.manual_seed(_seed(cfg.index, t, KIND_BIAS))
        rank = torch.randperm(cfg.E, generator=g)
        bias = (-1.2 * torch.log(rank.to(torch.float64) + 1.0)).to(torch.float32)
    else:
        bias = None
    return wr, bias


def group_weights(cfg: Config, t: int, e: int):
    """(W1 [d,f], W2 [f,d]) of expert e of task t, in the config's dtype."""
    w1 = _randn((cfg.d, cfg.f), _seed(cfg.index, t, KIND_W1, e), 1.0 / math.sqrt(cfg.d), "cpu")
    w2 = _randn((cfg.f, cfg.d), _seed(cfg.index, t, KIND_W2, e), 1.0 / math.sqrt(cfg.f), "cpu")
    return w1.to(cfg.torch_dtype), w2.to(cfg.torch_dtype)


def task_tokens(cfg: Config, t: int):
    """(x [N,d], dY [N,d]) of task t, in the config's dtype."""
    x = _randn((cfg.N, cfg.d), _seed(cfg.index, t, KIND_X), 1.0, "cpu")
    dy = _randn((cfg.N, cfg.d), _seed(cfg.index, t, KIND_DY), 1.0, "cpu")
    return x.to(cfg.torch_dtype), dy.to(cfg.torch_dtype)


def make_inputs(cfg: Config, device="cpu", tasks=None, with_weights=True):
    """All inputs of one step as a dict of tensors on ``device``.

    ``tasks`` selects a subset of task indices (default all), which regenerates
    exactly the same values those tasks get in the full problem.
    Keys: x [T,N,d], dy [T,N,d], w_router [T,d,E], bias [T,E] or None,
    w1 [T,E,d,f], w2 [T,E,f,d].
    """
    tasks = list(range(cfg.T)) if tasks is None else list(tasks)
    Tn = len(tasks)
    dt = cfg.torch_dtype
    x = torch.empty((Tn, cfg.N, cfg.d), dtype=dt, device=device)
    dy = torch.empty_like(x)
    wr = torch.empty((Tn, cfg.d, cfg.E), dtype=torch.float32, device=device)
    bias = None if cfg.bias == "none" else torch.empty((Tn, cfg.E), dtype=torch.float32,
                                                       device=device)
    w1 = w2 = None
    if with_weights:
        w1 = torch.empty((Tn, cfg.E, cfg.d, cfg.f), dtype=dt, device=device)
        w2 = torch.empty((Tn, cfg.E, cfg.f, cfg.d), dtype=dt, device=device)
    for i, t in enumerate(tasks):
        r, b = task_router(cfg, t)
        wr[i].copy_(r)
        if bias is not None:
            bias[i].copy_(b)
        xt, dyt = task_tokens(cfg, t)
        x[i].copy_(xt)
        dy[i].copy_(dyt)
        if with_weights:
            for e in range(cfg.E):
                a1, a2 = group_weights(cfg, t, e)
                w1[i, e].copy_(a1)
                w2[i, e].copy_(a2)
    return dict(x=x, dy=dy, w_router=wr, bias=bias, w1=w1, w2=w2)


def make_weights_fast(cfg: Config, device, seed: int = 0):
    """Weights of the right shape and distribution drawn directly on ``device``.

    Used where only throughput matters (the benchmark's timed run): it avoids
    generating gigabytes on the host.  Values differ from ``make_inputs``.
    """
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    dt = cfg.torch_dtype
    w1 = torch.randn((cfg.T, cfg.E, cfg.d, cfg.f), generator=g, device=device,
                     dtype=torch.float32).mul_(1.0 / math.sqrt(cfg.d)).to(dt)
    w2 = torch.randn((cfg.T, cfg.E, cfg.f, cfg.d), generator=g, device=device,
                     dtype=torch.float32).mul_(1.0 / math.sqrt(cfg.f)).to(dt)
    return w1, w2
