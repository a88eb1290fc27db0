"""bench.py's host-side contract: the reference arm's JSON line, the traffic gate and
the kernel label (no GPU needed)."""
import json
import os
import subprocess
import sys
import types

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402

BASE_KEYS = {"metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
             "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config"}


def test_reference_arm_prints_one_json_line():
    r = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--steps", "1",
                        "--warmup", "0"], cwd=ROOT, capture_output=True, text=True, timeout=600,
                       env=dict(os.environ, CUDA_VISIBLE_DEVICES=""))
    assert r.returncode == 0, r.stderr
    lines = [ln for ln in r.stdout.splitlines() if ln.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert BASE_KEYS <= set(d)
    assert d["impl"] == "reference" and d["metric"] == bench.METRIC and d["unit"] == bench.UNIT
    assert d["value"] > 0 and d["higher_is_better"] is True and d["steps"] == 1
    assert d["config"]["workload"] == "batch64-bf16-32L-32q8kv-d128-600u-off300-B4096-W10"
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["value"] == d["value"]
    assert d["cpu_baseline"]["cores"] >= 1 and d["cpu_baseline"]["sample"]
    e = d["e2e"]
    assert e["value"] == d["value"] and e["unit"] == d["unit"]
    assert e["h2d_bytes_per_step"] == 0 and e["d2h_bytes_per_step"] == 0


def test_traffic_is_reported_only_for_the_captured_sources(tmp_path, monkeypatch):
    import hashlib
    a, b = tmp_path / "a.cu", tmp_path / "b.cuh"
    a.write_text("int kernel(int x) { return x + 1; }  // a comment\n")
    b.write_text("/* header */ int y;\n")
    digest = hashlib.sha256(b"int kernel(int x) { return x + 1; }" + b"int y;").hexdigest()
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    monkeypatch.setattr(bench, "DECODE_TRAFFIC_SOURCES", ("a.cu", "b.cuh"))
    monkeypatch.setattr(bench, "DECODE_TRAFFIC_SHA256", digest)
    assert bench.decode_traffic(1000.0) == pytest.approx(1000.0 * bench.DECODE_TRAFFIC_RATIO)
    assert bench.decode_traffic(None) is None
    # comments and layout do not count ...
    a.write_text("int kernel(int x)\n{\n  return x + 1;  // another comment\n}\n")
    assert bench.decode_traffic(1000.0) == pytest.approx(1000.0 * bench.DECODE_TRAFFIC_RATIO)
    # ... code does
    a.write_text("int kernel(int x) { return x + 2; }\n")
    assert bench.decode_traffic(1000.0) is None


def test_the_committed_traffic_ratio_matches_the_committed_sources():
    """The ratio was taken on the decode sources as committed: the gate passes."""
    assert bench.decode_traffic(1.0e9) == pytest.approx(1.0e9 * bench.DECODE_TRAFFIC_RATIO)
    assert 1.0 <= bench.DECODE_TRAFFIC_RATIO < 1.05


@pytest.mark.parametrize("sessions,label", [
    (1, "attn_decode_split_kernel (16 warps)"),
    (3, "attn_decode_split_kernel (16 warps)"),
    (4, "attn_decode_split_kernel (4 warps)"),
    (9, "attn_decode_split_kernel (4 warps)"),
    (10, "attn_decode_split_kernel (4 warps)"),
    (19, "attn_decode_split_kernel (4 warps)"),
    (28, "attn_decode_split_kernel (4 warps)"),
    (57, "attn_decode_split_kernel (4 warps)"),
    (58, "attn_decode_kernel"),
    (64, "attn_decode_kernel"),
])
def test_roofline_kernel_label_follows_the_dispatch(sessions, label, monkeypatch):
    import torch
    monkeypatch.setattr(torch.cuda, "get_device_properties",
                        lambda i: types.SimpleNamespace(multi_processor_count=152))
    w = types.SimpleNamespace(n_sessions=sessions, kv_heads=8)
    assert bench.decode_kernel_label(w) == label
