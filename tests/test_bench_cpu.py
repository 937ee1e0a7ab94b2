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


@pytest.mark.parametrize("name", ["batch128", "hunyuan64", "solids96", "ring12_128", "tiny"])
def test_step_runs_cover_the_trajectory(name):
    """The bench's graphs: maximal runs of one kind of step, in order, covering
    every sampler step once; the build joins the first run exactly when the
    trajectory opens with a full step (the schedule from the oracle)."""
    import oracle
    w = synth.make_workload(name, B=1)
    cached = {t for t in range(w.S) if not oracle.is_full_step(t, w.S, w.schedule)}
    runs = bench.step_runs(w.S, cached)
    assert runs[0][0] == 0 and runs[-1][1] == w.S
    for (t0, u0, c0, _), (t1, u1, c1, _) in zip(runs, runs[1:]):
        assert u0 == t1 and c0 != c1
    for t, u, c, head in runs:
        assert t < u and all((k in cached) == c for k in range(t, u))
        assert head == (t == 0 and not c)
    assert runs[0][3] == (0 not in cached)
    if name == "batch128":  # a full step every fifth step: F CCCC x 6
        assert [(u - t, c) for t, u, c, _ in runs] == [(1, False), (4, True)] * 6
