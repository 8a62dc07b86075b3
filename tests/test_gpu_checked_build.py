"""The checked build (libfastrl_grpo_checked.so, build.py's checked=True): the same kernels with
GRPO_CHECKED defined test every index they compute before reading or writing through it (gathered
rows and rollouts, shared-memory layouts, the address, size and alignment of each asynchronous
copy, tile coordinates, output extents) and report a failure through grpo_debug_checks instead of
making the access.  It stands in for a device memory checker, which this GPU pool does not offer.

test_parity_suites_under_the_checked_build re-runs the GPU parity files in a child process with
FASTRL_GRPO_CHECKED=1: every test must pass there too, and conftest's autouse fixture asserts after
each one that no check fired.  The full-size workloads are left out (their time is the oracle's,
and their launch shapes are those of the smaller cases).  In that child process,
test_a_negative_row_index_is_caught feeds the loss a negative source row and a negative rollout id:
the checks replace them before any access (row 0, rollout 0) and report loss.cu.  That test runs
only under the checked build, whose checks precede every use of those two indices; the normal
build would read outside the caller's arrays."""
import os
import subprocess
import sys

import numpy as np
import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
FILES = ["tests/test_gpu_select.py", "tests/test_gpu_loss.py", "tests/test_gpu_logp.py",
         "tests/test_gpu_gspo.py", "tests/test_gpu_fuzz.py", "tests/test_gpu_pipeline.py",
         "tests/test_gpu_lmhead.py", "tests/test_gpu_lmhead_grad.py",
         "tests/test_gpu_sum.py", "tests/test_gpu_checked_build.py"]
LOSS_FILE_BIT = 3  # loss.cu in grpo_debug_checks' file mask


def test_parity_suites_under_the_checked_build():
    if os.environ.get("FASTRL_GRPO_CHECKED") == "1":
        pytest.skip("this process is the checked run")
    env = dict(os.environ, FASTRL_GRPO_CHECKED="1")
    r = subprocess.run([sys.executable, "-m", "pytest", *FILES, "-m", "gpu", "-q", "-x",
                        "-p", "no:cacheprovider", "-k", "not full_size"],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=2400)
    tail = r.stdout[-3000:] + r.stderr[-2000:]
    assert r.returncode == 0, tail
    assert " passed" in r.stdout.splitlines()[-1], tail
    print(r.stdout.splitlines()[-1])


@pytest.mark.expect_index_checks
def test_a_negative_row_index_is_caught(grpo):
    import torch
    if not grpo.checked_build():
        pytest.skip("only under the checked build (the child process of the test above)")
    assert b"checked" in grpo.lib().grpo_version()  # never the normal build: see the docstring
    grpo.grpo_debug_checks(reset=True)
    rng = np.random.default_rng(5)
    T, V = 40, 3000
    dev = "cuda"
    logits = torch.from_numpy(rng.normal(0, 2, (T, V)).astype(np.float32)).to(dev, torch.bfloat16)
    y = torch.from_numpy(rng.integers(0, V, T).astype(np.int32)).to(dev)
    old = torch.full((T,), -8.0, device=dev)
    ref = torch.full((T,), -8.1, device=dev)
    adv = torch.ones(4, device=dev)
    rollout = torch.from_numpy(np.repeat(np.arange(4, dtype=np.int32), 10)).to(dev)
    row_index = torch.arange(T, dtype=torch.int64, device=dev)
    row_index[5] = -3
    rollout[7] = -2
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    grpo.grpo_loss_fwd_bwd(logits, y, old, ref, adv, rollout, row_index=row_index, status=status)
    mask, site = grpo.grpo_debug_checks(reset=True)
    assert mask == 1 << LOSS_FILE_BIT and site // 100000 == LOSS_FILE_BIT, (mask, site)
    assert grpo.grpo_debug_checks(reset=True) == (0, 0)  # the record was cleared
