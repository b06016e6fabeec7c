"""bench.py's reference arm (the CPU oracle) prints one JSON line with the keys
the benchmark contract asks for; ranks other than 0 print nothing (no GPU)."""
import json
import os
import subprocess
import sys
from pathlib import Path

ROOT = Path(__file__).resolve().parent.parent


def _run(extra_env=None):
    env = dict(os.environ)
    env.update(extra_env or {})
    return subprocess.run([sys.executable, str(ROOT / "bench.py"), "--impl", "reference", "--steps", "2",
                           "--warmup", "3"], cwd=ROOT, env=env, capture_output=True, text=True, timeout=300)


def test_reference_arm_line():
    r = _run()
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference"
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
                "scaling", "vs_baseline", "dtype", "data", "config"):
        assert key in d, key
    assert d["value"] > 0 and d["unit"] == "tokens/s" and d["higher_is_better"] is True
    assert d["steps"] == 2 and d["warmup"] == 3 and d["n_gpus"] == 1
    assert d["vs_baseline"] is None
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["value"] == d["value"] and cb["cores"] >= 1 and cb["sample"]
    e2e = d["e2e"]
    assert e2e["value"] == d["value"] and e2e["unit"] == d["unit"]
    assert e2e["h2d_bytes_per_step"] == 0 and e2e["d2h_bytes_per_step"] == 0


def test_reference_arm_other_ranks_are_silent():
    r = _run({"RANK": "1", "WORLD_SIZE": "2"})
    assert r.returncode == 0, r.stderr[-2000:]
    assert r.stdout.strip() == ""


def test_bench_helpers():
    sys.path.insert(0, str(ROOT))
    import bench
    # the recorded DRAM traffic is reported only for the kernel source it was measured on
    recs = json.loads((ROOT / "profiles" / "traffic.json").read_text())["k_decode"]
    for workload in ("llama2-7b-block", "llama2-13b-block"):
        rec = recs[workload]
        got = bench.recorded_traffic("k_decode", "gs_decode.cu", workload)
        if rec["source_sha256_16"] == bench.kernel_source_hash("gs_decode.cu"):
            assert got == rec["dram_bytes_per_launch"]
        else:
            assert got is None
    assert bench.recorded_traffic("k_decode", "gs_decode.cu", "no-such-workload") is None
    assert bench.recorded_traffic("no_such_kernel", "gs_decode.cu", "llama2-7b-block") is None
    # threads kept busy = process CPU time / wall time, at least one
    assert bench._cores_used(30.0, 10.0) == 3 and bench._cores_used(0.2, 10.0) == 1
    assert bench._cores_used(5.0, 0.0) == 1


def test_single_thread_oracle_baseline():
    sys.path.insert(0, str(ROOT))
    import bench
    d = bench.oracle_single_thread_rate(0.5)
    assert "error" not in d, d
    assert d["cores"] == 1 and d["value"] > 0 and d["unit"] == "tokens/s" and d["sample"]
