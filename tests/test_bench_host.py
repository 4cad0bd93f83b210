"""Host-side logic of bench.py (no GPU): the reference arm's JSON line (the
CPU oracle timed on a bounded sample), its silence on ranks other than 0,
and the per-launch DRAM traffic taken from the committed ncu record."""
import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def _run(args, env_extra=None):
    env = dict(os.environ)
    env.update(env_extra or {})
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py")] + args, cwd=ROOT,
                       env=env, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    return r.stdout


def test_reference_arm_line():
    out = _run(["--impl", "reference", "--config", "1", "--steps", "2", "--warmup", "1",
                "--ref-total-s", "0.3"])
    lines = [l for l in out.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["unit"] == bench.UNIT and d["metric"] == bench.METRIC
    assert d["value"] > 0 and d["higher_is_better"] is True
    assert (d["steps"], d["warmup"], d["n_gpus"]) == (2, 1, 1)
    assert d["ms_per_step"] > 0
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == d["value"]
    assert "random locations" in cb["sample"]
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"], "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}
    # every location of configuration 1's 64 fits in the sample
    assert d["config"]["sample_locations_per_step"] == 64


def test_reference_arm_other_ranks_are_silent():
    out = _run(["--impl", "reference", "--config", "1", "--steps", "1", "--warmup", "0"],
               {"RANK": "1", "WORLD_SIZE": "2"})
    assert out.strip() == ""


def test_oracle_sampler_bounds():
    S = bench.OracleSampler(1, 2)
    k = S.calibrate(0.01)
    assert 1 <= k <= len(S.q)
    dt, m = S.run(k, seed=3)
    assert dt > 0 and m == min(k, len(S.q))


def test_traffic_record_scales_with_work():
    with open(os.path.join(ROOT, "profiles", "traffic.json")) as fh:
        rec = json.load(fh)
    for cls, r in rec.items():
        assert set(r) >= {"kernel", "dram_bytes", "alg_per_launch", "digest", "command"}
        assert r["command"].startswith("ncu ") and "--clock-control none" in r["command"]
        t1 = bench.traffic_per_launch(cls, r["alg_per_launch"])
        if t1 is None:   # the class's sources changed since the capture
            assert bench.sources_digest(cls) != r["digest"]
            continue
        assert t1 == pytest.approx(r["dram_bytes"])
        assert bench.traffic_per_launch(cls, 3 * r["alg_per_launch"]) == pytest.approx(3 * t1)
    assert bench.traffic_per_launch("no_such_class", 1.0) is None
