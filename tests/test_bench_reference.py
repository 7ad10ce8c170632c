"""bench.py's reference arm (the oracle on the host, no GPU): one JSON line
with the base contract's keys, the oracle's decode rate as `value` and
`cpu_baseline`, and its compress step timed separately."""
from __future__ import annotations

import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_reference_arm_line():
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                        "--workload", "latency-1k", "--steps", "2", "--warmup", "3"],
                       cwd=ROOT, stdout=subprocess.PIPE, stderr=subprocess.PIPE, text=True, timeout=300)
    assert r.returncode == 0, r.stderr
    lines = [l for l in r.stdout.splitlines() if l.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["steps"] == 2 and d["warmup"] == 3 and d["n_gpus"] == 1
    assert d["value"] > 0 and d["unit"] == "KV-tokens/s" and d["higher_is_better"] is True
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["value"] == d["value"]
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"], "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}
    assert d["compress"]["unit"] == "token-heads/s" and d["compress"]["value"] > 0
    assert "1088 tokens" in d["compress"]["sample"]
    # the value is the oracle on every host core; the one-thread figure beside it
    assert d["cpu_baseline"]["cores"] == len(os.sched_getaffinity(0))
    assert d["single_thread"]["cores"] == 1 and d["single_thread"]["value"] > 0
