"""Command lines that run without a GPU: the bench's reference arm (the CPU oracle) and the sweep
input generator's CLI contract (no GPU)."""
import json
import os
import subprocess
import sys
from pathlib import Path

ROOT = Path(__file__).resolve().parent.parent


def test_bench_reference_arm_json_line():
    """`bench.py --impl reference` prints one JSON line with the base contract's keys and the
    oracle's own cpu_baseline / e2e records (the oracle has no host-device copies)."""
    env = dict(os.environ, CUDA_VISIBLE_DEVICES="")
    out = subprocess.run([sys.executable, str(ROOT / "bench.py"), "--impl", "reference", "--steps", "1",
                          "--warmup", "0"], capture_output=True, text=True, env=env, timeout=600, check=True)
    lines = [l for l in out.stdout.splitlines() if l.strip().startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    for k in ("impl", "metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
              "scaling", "vs_baseline", "dtype", "data", "config", "cpu_baseline", "e2e"):
        assert k in d, k
    assert d["impl"] == "reference" and d["value"] > 0 and d["higher_is_better"] is True
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["value"] == d["value"]
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["e2e"]["value"] == d["value"]


def test_bench_cpu_baseline_record():
    """The bench's cpu_baseline record (all cores, one thread, the literal oracle on the
    50-request instance, the host CPU) on a small sample, without a GPU."""
    sys.path.insert(0, str(ROOT))
    import bench
    from paper_2508_14544_gb300 import workloads as W
    w = W.make_workload("c2", range(0, 1024, 32))
    d = bench.cpu_baseline(w, budget_s=0.5)
    assert d["kind"] == "oracle" and d["value"] > 0 and d["cores"] >= 1 and d["unit"] == bench.UNIT
    assert d["single_thread"]["value"] > 0 and d["literal_c1"]["value"] > 0
    assert isinstance(d["cpu"], str) and d["cpu"]
