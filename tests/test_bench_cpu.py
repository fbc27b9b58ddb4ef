"""CPU checks of bench.py: the reference arm's JSON line and the source hash
that keeps profiled DRAM counters attached to the kernel they were taken on."""
import json
import os
import shutil
import subprocess
import sys
import time

import bench

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_reference_arm_prints_one_contract_line():
    # one timed step of the oracle on this host (the whole batch: seconds)
    t0 = time.perf_counter()
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                        "--steps", "1", "--warmup", "3"],
                       capture_output=True, text=True, timeout=600, cwd=ROOT)
    wall = time.perf_counter() - t0
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
                "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config"):
        assert key in d, key
    assert d["impl"] == "reference" and d["steps"] == 1 and d["warmup"] == 3
    assert d["unit"] == "tokens/s" and d["higher_is_better"] is True and d["value"] > 0
    assert d["config"]["workload"] == "qwen_full_b64"
    # the same config keys as the GPU arm, and a step time that is measured:
    # the timed steps fit inside the run's own wall time
    wl = bench.WORKLOADS["qwen_full_b64"]
    assert d["config"] == bench.workload_config("qwen_full_b64", wl, bench.synth.QWEN, 1)
    assert d["config"]["batch"] == 64 and 100 < d["union"]["mean"] <= 128
    assert d["steps"] * d["ms_per_step"] * 1e-3 < wall
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["value"] == d["value"] and cb["cores"] >= 1
    assert isinstance(cb["sample"], str) and cb["sample"]
    e2e = d["e2e"]
    assert e2e["value"] == d["value"] and e2e["unit"] == d["unit"]
    assert e2e["h2d_bytes_per_step"] == 0 and e2e["d2h_bytes_per_step"] == 0


def test_source_hash_ignores_comments_and_whitespace_only(tmp_path, monkeypatch):
    csrc = tmp_path / "paper_2609_34117_gb300" / "csrc"
    csrc.mkdir(parents=True)
    for name in ("expert_ffn.cu", "common.cuh"):
        shutil.copy(os.path.join(ROOT, "paper_2609_34117_gb300", "csrc", name), csrc / name)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    base = bench.kernel_source_hash()
    f = csrc / "common.cuh"
    f.write_text(f.read_text() + "\n// a comment\n/* and a\n   block */\n\n   \n")
    assert bench.kernel_source_hash() == base
    f.write_text(f.read_text() + "constexpr int kAnotherConstant = 1;\n")
    assert bench.kernel_source_hash() != base
