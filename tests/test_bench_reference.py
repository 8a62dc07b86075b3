"""bench.py's reference arm (the fp64 oracle on the host cores) on the CPU: one JSON line with the
keys the bench contract names, for the token-level and GSPO losses and the output layer fused
with the loss; ranks other than 0 print nothing and exit 0."""
import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def run_bench(*args, env=None):
    e = dict(os.environ)
    e.update(env or {})
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), *args], cwd=ROOT, env=e,
                       capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    return [json.loads(l) for l in r.stdout.splitlines() if l.startswith("{")]


@pytest.mark.parametrize("loss", ["grpo", "gspo", "lmhead", "lmhead-gspo"])
def test_reference_arm_line(loss):
    extra = ("--hidden", "64") if loss.startswith("lmhead") else ()
    lines = run_bench("--impl", "reference", "--config", "tiny", "--loss", loss, "--steps", "2",
                      "--warmup", "1", *extra)
    assert len(lines) == 1
    d = lines[0]
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "higher_is_better",
              "scaling", "vs_baseline", "dtype", "data", "config", "cpu_baseline", "e2e"):
        assert k in d, k
    assert d["impl"] == "reference" and d["value"] > 0 and d["steps"] == 2
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] >= 1
    assert d["cpu_baseline"]["value"] == d["value"]
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"], "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}
    # the same config keys as the repo arm's line, the loss included
    assert d["config"]["loss"] == loss
    if loss.startswith("lmhead"):
        assert d["config"]["D"] == 64


def test_reference_arm_other_ranks_are_silent():
    assert run_bench("--impl", "reference", "--config", "tiny", "--steps", "1", "--warmup", "1",
                     env={"RANK": "1", "WORLD_SIZE": "2", "LOCAL_RANK": "1"}) == []
