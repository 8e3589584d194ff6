"""Host-side bookkeeping of bench.py (no GPU): the recorded ncu traffic is
reported only while the kernel sources hash to their capture-time value and
the shape matches, and the roofline peaks come from the measured file with
the stated fallback."""
import hashlib
import json
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def _sha(sources):
    h = hashlib.sha256()
    for f in sources:
        with open(os.path.join(bench.CSRC, f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def test_recorded_traffic_follows_the_source_hash():
    # Fresh captures are reported; after a kernel change the line reports null
    # until the traffic is captured again (the counters describe the old code).
    for kind, e in bench.NCU_TRAFFIC.items():
        expect = e["bytes"] if e["sha"] == _sha(e["sources"]) else None
        assert bench.ncu_traffic(kind, e["shape"]) == expect
        if e["bytes"] is not None:  # a recorded figure names the committed summary it comes from
            assert os.path.exists(os.path.join(ROOT, e["profile"].split(" ")[0]))


def test_traffic_is_null_for_another_shape_or_changed_sources(monkeypatch):
    e = bench.NCU_TRAFFIC["gemm"]
    other = tuple(x + 256 for x in e["shape"])
    assert bench.ncu_traffic("gemm", other) is None
    monkeypatch.setitem(bench.NCU_TRAFFIC, "gemm", dict(e, sha="0" * 16))
    assert bench.ncu_traffic("gemm", e["shape"]) is None


def test_peaks_measured_file_and_fallback(tmp_path, monkeypatch):
    p = bench.load_peaks()
    if os.path.exists(os.path.join(ROOT, "MEASURED_PEAKS.json")):
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            m = json.load(f)
        assert p["src"] == "measured" and p["hbm_gbs"] == float(m["hbm_gbs"])
        assert p["bf16_tflops"] == float(m["bf16_tflops"])
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    f = bench.load_peaks()
    assert f["src"] == "fallback" and f["hbm_gbs"] == 6800.0 and f["bf16_tflops"] == 1900.0
    (tmp_path / "MEASURED_PEAKS.json").write_text(json.dumps({"hbm_gbs": 7000, "bf16_tflops": 2000}))
    g = bench.load_peaks()
    assert g["src"] == "measured" and g["bf16_tflops_sustained"] == 2000.0


def test_gpus_flag_must_match_the_launched_world(monkeypatch):
    # --gpus N without N ranks would silently time one replica; it must fail.
    import subprocess
    env = dict(os.environ, WORLD_SIZE="1", RANK="0")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--gpus", "4", "--steps", "1"],
                       capture_output=True, text=True, env=env, timeout=120)
    assert r.returncode != 0 and "WORLD_SIZE=1" in r.stderr
