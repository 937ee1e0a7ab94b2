"""Host-side pieces of bench.py that need no GPU: the algorithmic byte count
of a cached step (12 B per element outside the anchor set, 16 B per anchor
element, bf16 latents) and the all-cores run of the CPU oracle (one spawned
process per share of the assets)."""
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2608_13255_gb300 import synth  # noqa: E402


def test_step_bytes_closed_form():
    w = synth.make_workload("batch128", B=2)
    per_asset = (4 * 12 + 2 * 16) * 4 * 128 * 128
    assert bench.step_bytes(w) == 2 * per_asset
    assert bench.step_bytes(w, 128) == 128 * per_asset == 671088640


def test_asset_subset_keeps_the_recipe():
    w = synth.make_workload("hunyuan64", B=1)
    w2 = synth.replicate_assets(w, 3)
    s = bench._asset_subset(w2, [1, 2])
    assert s.B == 2 and s.pos.shape[0] == 2 and s.cams.shape[0] == 2
    assert (s.name, s.S, s.a, s.schedule) == (w.name, w.S, w.a, w.schedule)


@pytest.mark.timeout(600)
def test_all_cores_oracle_baseline():
    w = synth.replicate_assets(synth.make_workload("hunyuan64", B=1), 2)
    r = bench.cpu_baseline_all_cores(w, cores=2)
    assert r["cores"] == 2 and r["kind"] == "oracle" and r["value"] > 0
    assert "all 2 assets" in r["sample"]


def test_reference_arm_prints_one_json_line():
    """`bench.py --impl reference` times the oracle (the reference arm) and
    prints the contract's keys; no GPU is touched."""
    import json
    import subprocess
    cmd = [sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--steps", "1", "--warmup", "1",
           "--workload", "hunyuan64", "--assets", "1", "--ref-assets", "1"]
    res = subprocess.run(cmd, capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert res.returncode == 0, res.stderr[-2000:]
    lines = [l for l in res.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["metric"] == bench.METRIC and d["unit"] == bench.UNIT
    assert d["value"] > 0 and d["higher_is_better"] is True and d["steps"] == 1
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] == 1
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["e2e"]["d2h_bytes_per_step"] == 0
