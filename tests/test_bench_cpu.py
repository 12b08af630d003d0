"""bench.py on the host: the reference arm's JSON line and the CPU-baseline helpers.

The reference arm times the fp64 oracle on the host cores (this tier has no
reference implementation to install); its line must carry the keys the bench
contract names.  No GPU is used.
"""
import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)


def test_reference_arm_prints_one_contract_line():
    res = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--steps", "3",
                          "--warmup", "1", "--workload", "tiny_p512_f4"],
                         cwd=ROOT, capture_output=True, text=True, timeout=300)
    assert res.returncode == 0, res.stderr
    lines = [ln for ln in res.stdout.splitlines() if ln.strip().startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference"
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
                "higher_is_better", "dtype", "config", "cpu_baseline", "e2e"):
        assert key in d, key
    assert d["value"] > 0 and d["steps"] == 3 and d["warmup"] == 1
    assert d["config"]["workload"] == "tiny_p512_f4"
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] >= 1
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["e2e"]["d2h_bytes_per_step"] == 0
    assert d["e2e"]["value"] == d["value"]


def test_oracle_children_and_cpu_model(monkeypatch):
    monkeypatch.setattr(sys, "argv", ["bench.py"])  # bench parses its arguments on import
    import bench
    assert bench.cpu_model()
    res = bench._oracle_children("tiny_p512_f4", 0.2, 2)
    assert len(res) == 2
    for forks, dt in res:
        assert forks >= 1 and dt > 0
    line = bench.cpu_baseline_all_cores("tiny_p512_f4", 0.2, 1 << 20)
    assert line["cores"] == min(16, os.cpu_count() or 1) and line["value"] > 0
    assert bench.cpu_baseline_all_cores("tiny_p512_f4", 0.2, 2 << 30) is None


def test_secondary_summaries_from_child_lines(monkeypatch):
    """The default line's `secondary` block: one child run per other configuration,
    summarised from the child's own JSON line; a child that fails is reported with
    its error instead of being dropped."""
    monkeypatch.setattr(sys, "argv", ["bench.py"])
    import bench
    calls = []

    class Done:
        def __init__(self, rc, out, err=""):
            self.returncode, self.stdout, self.stderr = rc, out, err

    def fake_run(cmd, **kw):
        calls.append(cmd)
        name = cmd[cmd.index("--workload") + 1]
        if name == "mla_p16k_f8":
            return Done(1, "", "RuntimeError: boom")
        line = {"value": 1.5, "unit": "tokens/s", "ms_per_step": 0.01, "kernels": {},
                "roofline": {"frac": 0.5}, "tensor_pipe_pct": None, "clocks": {},
                "e2e": {"value": 1.0}, "config": {"workload": name}}
        return Done(0, "noise\n" + json.dumps(line) + "\n")

    monkeypatch.setattr(bench.subprocess, "run", fake_run)
    out = bench.secondary_workloads(7, 3)
    assert set(out) == set(bench.SECONDARY) - {bench.ARGS.workload}
    assert out["fork_p8k_f8"]["value"] == 1.5 and out["fork_p8k_f8"]["e2e"] == 1.0
    assert out["fork_p8k_f8"]["config"]["workload"] == "fork_p8k_f8"
    assert "boom" in out["mla_p16k_f8"]["error"]
    for cmd in calls:  # same steps and warm-up, no CPU baseline, no recursion
        assert cmd[cmd.index("--steps") + 1] == "7" and cmd[cmd.index("--warmup") + 1] == "3"
        assert "--no-cpu-baseline" in cmd and "--no-secondary" in cmd
