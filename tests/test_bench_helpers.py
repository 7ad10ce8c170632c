"""bench.py's host-side helpers without a GPU: workload construction with its
overrides and range checks, the list of configurations the default run adds,
the per-workload summary, and the profile-traffic lookup's source-hash check."""
from __future__ import annotations

import os

import pytest

import bench


def test_make_workload_overrides_and_checks():
    wl = bench.make_workload("ksweep-32k", k_active=32)
    assert wl["k"] == 32 and wl["k_store"] == 128 and wl["k_v"] == 32 and wl["k_store_v"] == 128
    wl = bench.make_workload("llama2-7b-layer-32k", values="fp8_e4m3", k_store_v=32, batch=2)
    assert wl["values"] == "fp8_e4m3" and wl["k_store_v"] == 32 and wl["k_v"] == 32 and wl["B"] == 2
    assert wl["desc"] != bench.WORKLOADS["llama2-7b-layer-32k"]["desc"]   # the default run adds no workloads
    wl = bench.make_workload("basis-llama3-8b", tokens=4096)
    assert wl["n"] == 4096 and wl["k_v"] is None
    with pytest.raises(ValueError):
        bench.make_workload("llama2-7b-layer-32k", k_active=65)     # above k_store
    with pytest.raises(ValueError):
        bench.make_workload("llama2-7b-layer-32k", k_store_v=129)
    with pytest.raises(ValueError):
        bench.make_workload("llama2-7b-layer-32k", k_store_v=32, k_active_v=40)


def test_sub_workloads_cover_every_configuration():
    names = {name for _, name, _ in bench.SUB_WORKLOADS}
    # every workload appears (the headline's own with other value formats and
    # keep counts); the k sweep at each keep count
    assert names == set(bench.WORKLOADS)
    ks = sorted(over["k_active"] for _, name, over in bench.SUB_WORKLOADS if name == "ksweep-32k")
    assert ks == [32, 48, 64, 96, 128]
    labels = [label for label, _, _ in bench.SUB_WORKLOADS]
    assert len(labels) == len(set(labels))
    for _, name, over in bench.SUB_WORKLOADS:
        bench.make_workload(name, **over)       # each is a valid configuration


def test_summarize_keeps_the_figures_and_derives_the_70_percent_time():
    line = {"config": {"desc": "x", "l2": "inputs larger than L2"}, "value": 1.0, "unit": "KV-tokens/s",
            "ms_per_step": 2.0, "steps": 10, "warmup": 3, "gpu_launches": 20, "e2e": {"value": 0.5},
            "clocks": {"sm_mhz": 2070.0}, "prefill_ms": 8.0,
            "roofline": {"kernel": "decode", "bound": "hbm", "achieved": 6000.0, "peak": 6764.0, "unit": "GB/s",
                         "frac": 0.887, "pct_of_8tbs": 75.0, "alg_bytes_per_launch": 5.6e9,
                         "avg_launch_ms": 1.0, "traffic": None}}
    s = bench.summarize(line)
    assert s["roofline"]["frac"] == 0.887 and s["prefill_ms"] == 8.0 and s["e2e"] == {"value": 0.5}
    assert s["launch_ms_at_70pct_of_8tbs"] == pytest.approx(5.6e9 / (0.7 * 8000e9) * 1e3)
    line["config"]["l2"] = "L2 flushed (512 MB written) before every timed step"
    assert "launch_ms_at_70pct_of_8tbs" not in bench.summarize(line)    # latency, not a bandwidth


def test_profile_traffic_requires_matching_source_hashes(tmp_path, monkeypatch):
    # a profile whose hash line names the current source gives its traffic;
    # a stale hash, or a file it names that does not exist, gives None
    root = tmp_path
    (root / "profiles").mkdir()
    src = root / "paper_2511_18936_gb300" / "csrc"
    src.mkdir(parents=True)
    (src / "decode_kernels.cuh").write_text("// kernel source\n")
    import hashlib
    h = hashlib.sha256(b"// kernel source\n").hexdigest()[:16]
    monkeypatch.setattr(bench, "ROOT", str(root))
    (root / "profiles" / "decode_kernel_w.md").write_text(
        f"decode_kernels.cuh sha256[:16]: {h}\n\ndram bytes per launch: 1.5e9\n")
    assert bench.decode_kernel_traffic("w") == 1.5e9
    (root / "profiles" / "decode_kernel_w.md").write_text(
        "decode_kernels.cuh sha256[:16]: 0000000000000000\ndram bytes per launch: 1.5e9\n")
    assert bench.decode_kernel_traffic("w") is None
    (root / "profiles" / "decode_kernel_w.md").write_text(
        f"decode_kernels.cuh sha256[:16]: {h}, other.cuh sha256[:16]: {h}\ndram bytes per launch: 1.5e9\n")
    assert bench.decode_kernel_traffic("w") is None
    assert bench.decode_kernel_traffic("missing") is None


def test_host_cores_is_the_affinity_set():
    assert bench.host_cores() == len(os.sched_getaffinity(0))


def test_committed_profiles_are_reproducible_summaries():
    # every ncu command a summary gives leaves the clocks alone, names only
    # committed entry points, and every kernel file a summary hashes exists
    import glob
    import re
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    files = glob.glob(os.path.join(root, "profiles", "*.md"))
    assert files
    for path in files:
        text = open(path).read()
        cmds = re.findall(r"^[ \t]*ncu (?:[^\n]*\\\n)*[^\n]*", text, flags=re.M)
        assert cmds, path
        for cmd in cmds:
            assert "--clock-control none" in cmd, (path, cmd)
            assert "_work" not in cmd, (path, cmd)
            assert re.search(r"python (bench\.py|-c)", cmd), (path, cmd)
        for name in re.findall(r"([\w.]+\.(?:cuh|cu)) sha256\[:16\]", text):
            assert os.path.exists(os.path.join(root, "paper_2511_18936_gb300", "csrc", name)), (path, name)
