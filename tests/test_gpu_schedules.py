"""The library's optional schedules, each switched on by an environment variable
that it reads once per process, run the GPU parity tests again in a child process:

  VMOE_ROW_PAIR=1  row-mode GEMMs of groups above 128 rows on SM pairs (256-row
                   tiles): the capacity-256 group-tail cases, against the oracle
                   and sliced against full, bitwise;
  VMOE_SHARES=1    the memory-budgeted backward's dW1 with each group's column
                   tiles on a share of the SM pairs from the fill-clamp-refill
                   allocation (Section 3.2.2): the sliced-backward cases, which
                   must stay bitwise equal to the unsliced backward, and the
                   group-tail cases.
  VMOE_ROUTE_TC=1  the tcgen05 router in place of the mma.sync one for bf16
                   tokens: the small parity cases (E = 4 to 16), the identity-
                   expert invariant and the 17-task ViT-B routing at full size
                   (E = 32).
"""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import __graft_entry__
    __graft_entry__.build()


def _child(env_name, targets, value="1"):
    env = dict(os.environ, **{env_name: value})
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-p", "no:cacheprovider", *targets],
                       cwd=os.path.dirname(HERE), env=env, capture_output=True, text=True, timeout=900)
    assert r.returncode == 0, r.stdout[-3000:] + r.stderr[-2000:]
    return r.stdout


def test_row_pair_schedule():
    out = _child("VMOE_ROW_PAIR", ["tests/test_gpu_tails.py::test_group_tails[bf16-512-256-256]",
                                   "tests/test_gpu_tails.py::test_group_tails[bf16-384-640-256]"])
    assert "2 passed" in out


def test_share_schedule():
    out = _child("VMOE_SHARES", ["tests/test_gpu_sliced_bwd.py",
                                 "tests/test_gpu_tails.py::test_group_tails[bf16-256-512-128]",
                                 "tests/test_gpu_tails.py::test_group_tails[bf16-512-256-256]"])
    assert "passed" in out and "failed" not in out


def test_tcgen05_router():
    out = _child("VMOE_ROUTE_TC", ["tests/test_gpu_parity.py::test_step_parity_small",
                                   "tests/test_gpu_parity.py::test_identity_experts_dispatch_combine",
                                   "tests/test_gpu_fullsize.py::test_fullsize_sampled_parity[vitb_t17]"])
    assert "passed" in out and "failed" not in out
