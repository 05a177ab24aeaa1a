"""bench.py on the CPU.  The reference arm (the fp64 oracle on the host cores) prints
one JSON line with the fields the bench contract requires: the same metric,
unit and direction as the GPU arm, its own e2e with no host-device traffic,
and a cpu_baseline describing the run (kind oracle, cores, sample, CPU).  The
roofline numerators of the five workloads match their shapes."""

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


# Algorithmic work per steady step of the five workloads, written out from
# their shapes (X and labels of the distinct evaluated partitions read once;
# the tensor-core contraction's 2 rows d K flops): the numerators of every
# roofline fraction bench.py reports.
EXPECTED_WORK = {
    "fr_n4_logistic_d64": ("hbm", 2 * 256 * (64 * 4 + 4)),                  # FR: n/c = 2 partitions
    "cr_n8_logistic_d1024": ("hbm", 8 * 8192 * (1024 * 4 + 4)),              # 268,697,600 B
    "fr_n32_softmax_k10": ("hbm", 8 * 4096 * (3072 * 2 + 4)),                # 201,457,664 B
    "cr_n64_lsq_d16384": ("hbm", 64 * 2048 * (16384 * 4 + 4)),               # 8,590,458,880 B
    "cr_n128_softmax_k1000": ("tensor", 2.0 * 128 * 1024 * 4096 * 1000),      # 1.074 TFLOP per contraction
}


@pytest.mark.parametrize("name", list(EXPECTED_WORK))
def test_roofline_numerators(name):
    from paper_2607_20739_gb300 import workloads as W
    bound, units, unit, peak = bench.roofline_model(W.WORKLOADS[name], {"hbm_gbs": 6784.8,
                                                                        "bf16_tflops_sustained": 1718.2})
    want_bound, want_units = EXPECTED_WORK[name]
    assert bound == want_bound
    assert units == pytest.approx(want_units, rel=0, abs=0.5)
    assert peak == (6784.8 if bound == "hbm" else 1718.2)
    assert unit == ("GB/s" if bound == "hbm" else "TFLOP/s")


def test_source_hash_ignores_comments_only(tmp_path, monkeypatch):
    d = tmp_path / "paper_2607_20739_gb300" / "csrc"
    d.mkdir(parents=True)
    f = d / "k.cu"
    f.write_text('// header\n__global__ void k(int* p) { p[0] = 1; /* one */ }\nconst char* s = "a//b";\n')
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    h0 = bench.kernel_source_hash()
    f.write_text('// header, reworded\n// over two lines\n__global__ void k(int* p) {\n  p[0] = 1;  // one\n}\n'
                 'const char* s = "a//b";\n')
    assert bench.kernel_source_hash() == h0
    f.write_text('__global__ void k(int* p) { p[0] = 2; }\nconst char* s = "a//b";\n')
    assert bench.kernel_source_hash() != h0
    f.write_text('__global__ void k(int* p) { p[0] = 1; }\nconst char* s = "a/*b";\n')
    assert bench.kernel_source_hash() != h0          # a comment marker inside a string is code
