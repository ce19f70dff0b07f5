"""HostPipeline: steps from pinned host buffers with the copies overlapped with
compute must give, step by step, exactly the outputs of the plain in-order
StepRunner on the same inputs (the pipeline only reorders copies, never compute).
"""
import pytest
import torch

import workloads
from gpu_helpers import problem_of, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import __graft_entry__
    __graft_entry__.build()


def test_pipeline_matches_in_order_steps():
    import paper_2608_16188_gb300 as vm
    cfg = workloads.Config("pipe", 70, T=3, N=197, d=256, f=512, E=4, k=2, cf=1.25, dtype="bf16",
                           bias="drift")
    inp = to_dev(workloads.make_inputs(cfg))
    p = problem_of(cfg)
    steps = 5
    g = torch.Generator().manual_seed(3)
    xs = [(torch.randn(inp["x"].shape, generator=g).to(torch.bfloat16).pin_memory(),
           torch.randn(inp["dy"].shape, generator=g).to(torch.bfloat16).pin_memory())
          for _ in range(steps)]
    outs = [(torch.empty(inp["x"].shape, dtype=torch.bfloat16).pin_memory(),
             torch.empty(inp["x"].shape, dtype=torch.bfloat16).pin_memory()) for _ in range(steps)]
    weights = {k: v for k, v in inp.items() if k not in ("x", "dy")}
    pipe = vm.HostPipeline(p, weights, device="cuda")
    pipe.run(xs, outs)
    torch.cuda.synchronize()
    ref = vm.StepRunner(p, dict(inp))
    for i in range(steps):
        ref.inp["x"].copy_(xs[i][0])
        ref.inp["dy"].copy_(xs[i][1])
        ref.step()
        torch.cuda.synchronize()
        assert torch.equal(outs[i][0], ref.b.y.cpu()), i
        assert torch.equal(outs[i][1], ref.b.dx.cpu()), i
    assert vm.vmoe_device_status() == 0
