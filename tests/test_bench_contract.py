"""bench.py's reference arm (CPU only): ``--impl reference`` runs the oracle on
the host cores and prints one JSON line with the GPU arm's metric, unit and
workload keys, the oracle's own cpu_baseline, a host-only e2e, and a
ms_per_step that is the time of one batch-32 full-vocabulary step at the
measured rate."""
import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_reference_arm_line():
    sys.path.insert(0, ROOT)
    import bench
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--steps", "1",
                          "--warmup", "0", "--ref-tokens", "1024"], capture_output=True, text=True, timeout=600,
                         cwd=ROOT)
    assert out.returncode == 0, out.stderr[-2000:]
    line = json.loads(out.stdout.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["metric"] == bench.METRIC and line["unit"] == "masks/s"
    assert line["higher_is_better"] is True and line["steps"] == 1 and line["warmup"] == 0
    assert line["config"] == bench.headline_config(32, 151936)
    v = line["value"]
    assert v > 0 and abs(line["ms_per_step"] - 32 / v * 1e3) <= 1e-6 * line["ms_per_step"]
    cb = line["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == v and cb["unit"] == "masks/s" and cb["sample"]
    assert line["e2e"] == {"value": v, "unit": "masks/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}
    assert line["vs_baseline"] is None
