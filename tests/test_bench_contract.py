"""bench.py's JSON line, checked without a GPU: the reference arm (the oracle on the
host cores) run end to end on a tiny sample, and the workload description both arms
share.  The GPU arm's own line is produced on the GPU machine only."""
import json
import os
import subprocess
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)


def test_reference_arm_prints_one_complete_line():
    p = subprocess.run(
        [sys.executable, "bench.py", "--impl", "reference", "--steps", "2", "--warmup", "0",
         "--workload", "llama", "--cpu-units", "1", "--cpu-rows", "256"],
        cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert p.returncode == 0, p.stderr[-2000:]
    lines = [l for l in p.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, p.stdout
    d = json.loads(lines[0])
    for k, t in [("metric", str), ("value", float), ("unit", str), ("n_gpus", int),
                 ("steps", int), ("warmup", int), ("ms_per_step", float),
                 ("higher_is_better", bool), ("scaling", str), ("dtype", str), ("data", str),
                 ("config", dict), ("impl", str), ("cpu_baseline", dict), ("e2e", dict)]:
        assert isinstance(d[k], t), k
    assert d["impl"] == "reference" and d["n_gpus"] == 1 and d["steps"] == 2
    assert d["vs_baseline"] is None and d["higher_is_better"] is True
    assert d["value"] > 0 and d["ms_per_step"] > 0
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["sample"]
    assert cb["value"] == d["value"] and cb["unit"] == d["unit"]
    e = d["e2e"]
    assert e["value"] == d["value"] and e["unit"] == d["unit"]
    assert e["h2d_bytes_per_step"] == 0 and e["d2h_bytes_per_step"] == 0
    c = d["config"]
    assert c["L"] == 16 and c["H"] == 8 and c["N"] == 8192 and c["d"] == 64
    assert "Llama-3.2-1B" in c["workload"]


@pytest.mark.parametrize("schedule", ["uniform", "pyramid"])
@pytest.mark.parametrize("path", ["repair", "dedup", "policy"])
def test_workload_config(schedule, path):
    import bench
    from paper_2608_27128_gb300 import synth
    w = synth.get("qwen")
    c = bench.workload_config(w, 0.5, path, schedule)
    assert c["path"] == path and c["schedule"] == schedule
    assert (c["L"], c["H"], c["N"], c["d"]) == (36, 8, 16384, 128)
    assert c["tau"] == 0.85 and c["window"] == 32 and c["n_sink"] == 4 and c["n_recent"] == 64
    assert "no flush" in c["l2"] and c["parallelism"] == "replicas"
    if schedule == "pyramid":
        k = c["budget_per_layer"]
        assert len(k) == 36 and sum(k) == 36 * synth.budget(w, 0.5)
        assert "pyramid" in c["workload"]
    else:
        assert c["budget_per_layer"] is None


def test_traffic_record_matches_the_audit_sources():
    """The committed DRAM-traffic record is keyed to the audit kernel's sources; when
    they match, a full launch's traffic scales with the units."""
    import bench
    t1 = bench.audit_traffic(1)
    if t1 is None:
        pytest.skip("audit sources changed since the traffic capture")
    assert bench.audit_traffic(288) == pytest.approx(288 * t1)
    # about the algorithmic bytes of one unit (keys as A and B, metadata): 8.7 MB
    assert 8.0e6 < t1 < 9.5e6
