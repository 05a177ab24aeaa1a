"""The reference arm of bench.py (the fp64 oracle on the host cores) prints
one JSON line with the fields the bench contract requires: the same metric,
unit and direction as the GPU arm, its own e2e with no host-device traffic,
and a cpu_baseline describing the run (kind oracle, cores, sample, CPU)."""

import json
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402

REQUIRED = ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better", "scaling",
            "vs_baseline", "dtype", "data", "config", "impl", "cpu_baseline", "e2e")


@pytest.mark.parametrize("mode", ["pgc", "naive_cr"])
def test_reference_line_fields(capsys, monkeypatch, mode):
    for k in ("RANK", "WORLD_SIZE", "LOCAL_RANK"):
        monkeypatch.delenv(k, raising=False)
    workload = "fr_n4_logistic_d64" if mode == "pgc" else "cr_n8_logistic_d1024"
    args = bench.parse_args(["--impl", "reference", "--workload", workload, "--mode", mode, "--steps", "2",
                             "--warmup", "3", "--cpu-seconds", "0.5"])
    bench.run_reference(args)
    lines = [l for l in capsys.readouterr().out.splitlines() if l.strip().startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    for k in REQUIRED:
        assert k in d, k
    assert d["impl"] == "reference" and d["metric"] == bench.METRIC and d["unit"] == "steps/s"
    assert d["higher_is_better"] is True and d["n_gpus"] == 1 and d["vs_baseline"] is None
    assert d["value"] > 0 and d["ms_per_step"] == pytest.approx(1000.0 / d["value"])
    assert d["config"]["workload"] == workload and d["config"]["mode"] == mode
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["value"] == d["value"] and cb["cores"] >= 1
    assert cb["sample"] and cb["cpu_model"]
    e = d["e2e"]
    assert e["value"] == d["value"] and e["unit"] == d["unit"]
    assert e["h2d_bytes_per_step"] == 0 and e["d2h_bytes_per_step"] == 0
