"""bench.py's output contract, checked without a GPU: the reference arm
(the oracle timed on the host cores) prints one JSON line with the keys the
measurement contract names, and the helpers that label a line's projection
kernel and attach a capture's DRAM traffic pick the right kernel and path."""
import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_reference_arm_prints_one_contract_line():
    r = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--workload", "tiny_b1",
                        "--steps", "1", "--warmup", "3"], cwd=ROOT, capture_output=True, text=True,
                       timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.strip().startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
              "scaling", "vs_baseline", "dtype", "data", "config", "cpu_baseline", "e2e"):
        assert k in d, k
    assert d["impl"] == "reference" and d["value"] > 0 and d["warmup"] >= 3 and d["steps"] == 1
    assert d["higher_is_better"] is True and d["config"]["workload"] == "tiny_b1"
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["value"] == d["value"] and cb["cores"] >= 1 and cb["sample"]
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"], "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}


def test_projection_labels_and_traffic_follow_the_path():
    sys.path.insert(0, ROOT)
    import bench
    assert bench._proj_kernel("skinny", 9).startswith("skinny_kernel")
    assert bench._proj_kernel("skinny", 144).startswith("skinny_mt_kernel")
    assert bench._proj_kernel("tcgen05", 9).startswith("gemm_tc_kernel")
    # a capture's traffic describes only the path it ran
    assert bench._gemm_traffic("large_b1", "skinny") == bench.GEMM_DRAM_BYTES_PER_LAUNCH["large_b1"]
    assert bench._gemm_traffic("large_b1", "tcgen05") is None
    assert bench._gemm_traffic("large_b16", "tcgen05") is None
    assert bench._gemm_traffic("large_b96", "tcgen05") == bench.GEMM_DRAM_BYTES_PER_LAUNCH["large_b96"]
    assert bench._gemm_traffic("tiny_b1", "skinny") is None
