"""bench.py is a one-GPU program: with --gpus other than 1, or started as one
of several ranks, the GPU arm stops with an error before torch (and so any
CUDA call) is loaded; the reference arm, which uses no GPU, runs on rank 0
only and prints nothing on the other ranks."""

import io
import json
import os
import subprocess
import sys
from contextlib import redirect_stdout

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402

PROBE = ("import sys, bench\n"
         "args = bench.parse_args(sys.argv[1:])\n"
         "try:\n"
         "    bench.run_ours(args)\n"
         "except SystemExit as e:\n"
         "    print('exit', e.code, 'torch' in sys.modules)\n")


def _probe(argv, env_extra):
    env = {k: v for k, v in os.environ.items() if k not in ("RANK", "WORLD_SIZE", "LOCAL_RANK")}
    env.update(env_extra)
    r = subprocess.run([sys.executable, "-c", PROBE, *argv], cwd=ROOT, env=env, capture_output=True, text=True,
                       timeout=120)
    assert r.returncode == 0, r.stderr
    return r.stdout.strip().splitlines()[-1], r.stderr


def test_more_than_one_gpu_is_refused_before_any_cuda_call():
    out, err = _probe(["--gpus", "2", "--steps", "2", "--warmup", "3"], {})
    assert out == "exit 2 False"                     # SystemExit(2), torch never imported
    msg = json.loads(err.strip().splitlines()[-1])
    assert msg["gpus"] == 2 and "one GPU" in msg["error"]


def test_a_multi_rank_launch_is_refused_on_every_rank():
    for rank in ("0", "1"):
        out, err = _probe(["--steps", "2"], {"RANK": rank, "WORLD_SIZE": "2", "LOCAL_RANK": rank})
        assert out == "exit 2 False"
        assert json.loads(err.strip().splitlines()[-1])["world_size"] == 2


def test_reference_arm_runs_on_rank_zero_only(monkeypatch):
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    monkeypatch.setenv("LOCAL_RANK", "1")
    args = bench.parse_args(["--impl", "reference", "--gpus", "2", "--steps", "2", "--warmup", "3"])
    out = io.StringIO()
    with redirect_stdout(out):
        bench.run_reference(args)
    assert out.getvalue() == ""
