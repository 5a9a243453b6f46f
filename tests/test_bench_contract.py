"""bench.py's output contract: one JSON line with the keys the benchmark
driver reads. The reference arm (the oracle on the host cores) runs here on
CPU; the GPU arm runs on a small workload under the gpu marker."""
import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _run(args, timeout=600):
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), *args], cwd=ROOT,
                       capture_output=True, text=True, timeout=timeout)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, r.stdout[-2000:]
    return json.loads(lines[0])


BASE_KEYS = ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
             "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config", "e2e",
             "gpu_launches")


def test_reference_arm_line():
    d = _run(["--impl", "reference", "--steps", "1", "--warmup", "1"])
    for k in BASE_KEYS + ("impl", "cpu_baseline"):
        assert k in d, k
    assert d["impl"] == "reference" and d["value"] > 0 and d["gpu_launches"] == 0
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["value"] == d["value"]
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"], "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}
    assert d["config"]["workload"] == "stress"


@pytest.mark.gpu
def test_gpu_arm_line():
    d = _run(["--workload", "tiny", "--steps", "5", "--warmup", "3", "--cpu-samples", "1",
              "--e2e-steps", "2"])
    for k in BASE_KEYS + ("roofline", "cpu_baseline", "clocks"):
        assert k in d, k
    assert d["value"] > 0 and d["n_gpus"] == 1 and d["steps"] == 5 and d["warmup"] == 3
    r = d["roofline"]
    for k in ("bound", "achieved", "peak", "unit", "frac", "traffic"):
        assert k in r, k
    assert r["bound"] == "hbm" and r["achieved"] > 0 and r["peak"] > 0
    assert d["gpu_launches"] >= d["steps"]
    assert d["e2e"]["h2d_bytes_per_step"] > 0 and d["e2e"]["d2h_bytes_per_step"] > 0
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] >= 1
    for k in ("sm_mhz", "sm_max_mhz", "reasons"):
        assert k in d["clocks"], k
    assert d["config"]["workload"] == "tiny"
    rows = d["next_rows"]
    for k in ("select_raw", "select_cache", "decode_1x933", "revisit_k32_graph"):
        assert k in rows, k
    assert rows["select_raw"]["ms"] > 0 and rows["select_cache"]["gbs"] > 0
    assert rows["decode_1x933"]["us"] > 0 and rows["revisit_k32_graph"]["us"] > 0


@pytest.mark.gpu
@pytest.mark.parametrize("path", ["capture", "decode", "select", "pipeline"])
def test_gpu_other_paths_line(path):
    """The capture, decode, selection and pipeline bench paths print one
    well-formed line each; the first three time the oracle beside the kernel."""
    args = ["--path", path, "--workload", "tiny", "--steps", "3", "--warmup", "3"]
    d = _run(args)
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
              "higher_is_better", "config", "gpu_launches", "clocks"):
        assert k in d, (path, k)
    assert d["value"] > 0 and d["gpu_launches"] >= d["steps"]
    if path != "pipeline":
        assert d["roofline"]["bound"] == "hbm" and d["roofline"]["achieved"] > 0
        c = d["cpu_baseline"]
        assert c["kind"] == "oracle" and c["cores"] == 1 and c["value"] > 0 and c["sample"]
