"""Host-side logic of bench.py, on the CPU: the timing percentiles, the
traffic figures that go stale with their kernel's sources, the BLAS thread
limiter the single-thread oracle timing uses, and the reference arm, which
runs whole oracle steps and reports how many it ran."""

import json
import os
import subprocess
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def test_percentiles_nearest_rank():
    per = [float(x) for x in range(1, 101)]        # 1 .. 100 ms
    p = bench.percentiles(per)
    assert p["ms_p50"] in (50.0, 51.0)
    assert p["ms_p10"] in (10.0, 11.0)
    assert p["ms_p90"] in (90.0, 91.0)
    assert bench.percentiles([3.0]) == {"ms_p10": 3.0, "ms_p50": 3.0, "ms_p90": 3.0}


def test_traffic_goes_stale_with_its_sources(tmp_path, monkeypatch):
    for key, e in bench.TRAFFIC.items():
        assert bench.traffic_of(*key) in (e["bytes"], None), key
    src = tmp_path / "k.cu"
    src.write_text("// kernel\n")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    monkeypatch.setitem(bench.TRAFFIC, ("k", "w"), {"bytes": 7, "sources": ["k.cu"],
                                                   "sha256": bench.sources_sha256(["k.cu"])})
    assert bench.traffic_of("k", "w") == 7
    src.write_text("// kernel, changed\n")
    assert bench.traffic_of("k", "w") is None
    assert bench.traffic_of("absent", "w") is None


def test_blas_threads_limits_and_restores():
    apis = bench._openblas_thread_apis()
    before = [g() for _, g in apis]
    with bench.blas_threads(1):
        a = np.ones((64, 64))
        assert float((a @ a)[0, 0]) == 64.0
        if apis:
            assert all(g() == 1 for _, g in apis)
    assert [g() for _, g in apis] == before


def test_reference_arm_reports_steps_it_ran():
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                          "--config", "tiny_f32", "--steps", "2", "--warmup", "1"],
                         capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert out.returncode == 0, out.stderr[-2000:]
    line = json.loads([x for x in out.stdout.splitlines() if x.startswith("{")][-1])
    assert line["impl"] == "reference" and line["steps"] == 2 and line["steps_requested"] == 2
    assert line["ms_per_step"] * line["steps"] / 1000.0 <= line["wall_s"]
    assert line["ms_p10"] <= line["ms_p50"] <= line["ms_p90"]
    cb = line["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["cpu_model"]
    assert line["e2e"]["h2d_bytes_per_step"] == 0
