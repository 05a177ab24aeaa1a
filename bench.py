#!/usr/bin/env python
"""Throughput of the PGC hot path on one GB300: one JSON line on stdout.

A "step" is one ``pgc_step`` call: every scheduled per-partition gradient,
the gradient-store commit, and the decode fused with the SGD update, over the
workload's resident partitions.  ``value`` is steady-state steps/s measured
with CUDA events on the library's stream (inputs resident in HBM).  ``e2e`` is
the same metric through the Python API with host buffers: the straggler mask
goes host->device and the decoded gradient and the new parameters come back
device->host every step.

  python bench.py [--steps K] [--warmup W]          # headline + every workload
  python bench.py --workload NAME [--override k=v]  # one workload only
  python bench.py --impl reference ...              # the fp64 CPU oracle

By default the headline line is the largest workload, cr_n128_softmax_k1000
(CR, n=128, s=7, softmax K=1000, d=4096), timed over exactly K steps, and
``per_workload`` carries the same fields for the other four workloads,
measured in the same invocation.  The simulated cluster lives on one GPU:
there is no multi-GPU form, so ``--gpus`` other than 1, or a launch with
several ranks, stops with an error before any CUDA call.
"""

from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2607_20739_gb300 import workloads as W  # noqa: E402

METRIC = "PGC steps/s & samples/s at 1 GB300; % of HBM (or bf16 TC) roofline"
HEADLINE_WORKLOAD = "cr_n128_softmax_k1000"   # the largest workload that fits one GPU
L2_BYTES = 129 * 2 ** 20
GC_DRAWS_SEED = 2607          # seed of the GC-CR encoding draws (naive_cr, and gc on CR placement)


def parse_args(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=None)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default=None, choices=W.WORKLOAD_ORDER,
                    help="measure this workload only (default: the headline workload, then every other one)")
    ap.add_argument("--no-per-workload", action="store_true", help="measure the headline workload only")
    ap.add_argument("--seed", type=int, default=1)
    ap.add_argument("--mode", default="pgc", choices=["pgc", "is_sgd", "gc", "naive_cr"],
                    help="training scheme on the same kernels: PGC, or the IS-SGD / GC (FR) baselines")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=15.0, help="budget of the oracle sample")
    ap.add_argument("--override", action="append", default=[],
                    help="KEY=VALUE change of the workload (n, s, m, d, K) for profiling smaller cases")
    return ap.parse_args(argv)


def workload_from_args(args) -> W.Workload:
    w = W.WORKLOADS[args.workload or HEADLINE_WORKLOAD]
    kw = {}
    for o in args.override:
        k, v = o.split("=", 1)
        if k not in ("n", "s", "m", "d", "K"):
            raise SystemExit(f"cannot override {k}")
        kw[k] = int(v)
    if kw:
        w = w.replace(name=w.name + "+" + ",".join(f"{k}={v}" for k, v in sorted(kw.items())), **kw)
    return w


# ---------------------------------------------------------------------------
# algorithmic work (per steady step)
# ---------------------------------------------------------------------------

def evaluated_rows(w: W.Workload) -> int:
    """Distinct rows evaluated per steady step: FR computes one partition per
    group (n/c partitions), CR all n."""
    rows = w.rows()
    if w.scheme == "FR":
        return sum(rows[g * w.c] for g in range(w.n // w.c))
    return sum(rows)


def grad_bytes_per_row(w: W.Workload) -> int:
    esz = 2 if w.dtype == "bf16" else 4
    return w.d * esz + 4


TC_MIN_CLASSES = 128          # the library runs bf16 softmax from this many classes on the tensor cores


def tensor_core_path(w: W.Workload) -> bool:
    return w.loss == "softmax" and w.dtype == "bf16" and TC_MIN_CLASSES <= w.K <= 2048


def roofline_model(w: W.Workload, peaks: dict):
    """(bound, algorithmic units per launch of the dominant kernel, unit, peak).

    Streaming paths: the gradient kernel reads the evaluated partitions' X and
    labels once (bytes).  Tensor-core softmax: each of the two GEMMs (logits
    X W^T and gradient R^T X) performs 2 rows d K flops per step; the slower
    of the two is reported."""
    rows = evaluated_rows(w)
    if tensor_core_path(w):
        flops = 2.0 * rows * w.d * w.K
        return "tensor", flops, "TFLOP/s", peaks.get("bf16_tflops_sustained") or 1700.0
    return "hbm", float(rows * grad_bytes_per_row(w)), "GB/s", peaks.get("hbm_gbs") or 6800.0


def kernel_label(w: W.Workload, single: bool, dom: int) -> str:
    if tensor_core_path(w):
        nt = -(-w.K // 256)
        if dom == 2:
            return "tc_grad_kernel, gradient R^T X (tcgen05.mma.cta_group::2 over CTA pairs, runs of partitions)"
        if nt in (1, 2, 4, 8):
            return f"tc_logits_softmax_kernel, logits X W^T + softmax residual (tcgen05, {nt}-CTA clusters)"
        return "tc_gemm_kernel, logits X W^T (tcgen05, 2-CTA clusters)"
    if w.loss == "softmax" and w.dtype == "bf16" and w.K <= 16:
        if -(-w.d // 128) * 128 <= 3072:
            return "softmax_rows_kernel (16-row tiles split by features over CTA pairs, one pass over X; whole step)"
        return "softmax_smallk_kernel (8-CTA clusters, one pass over X)"
    if w.loss == "softmax":
        return "CUDA-core softmax gradient kernels"
    return "grad_rows kernel with fused commit+decode (whole step)" if single else "grad_rows kernel"


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}, "fallback"


def _strip_comments(src: str) -> str:
    """C/C++ source without its // and /* */ comments (string and character
    literals kept), so that a comment-only edit leaves the hash unchanged."""
    out, i, n = [], 0, len(src)
    while i < n:
        ch = src[i]
        if ch in "\"'":
            j = i + 1
            while j < n and src[j] != ch:
                j += 2 if src[j] == "\\" else 1
            out.append(src[i:j + 1])
            i = j + 1
        elif src.startswith("//", i):
            j = src.find("\n", i)
            i = n if j < 0 else j
        elif src.startswith("/*", i):
            j = src.find("*/", i + 2)
            i = n if j < 0 else j + 2
        else:
            out.append(ch)
            i += 1
    return "".join(out)


def kernel_source_hash() -> str:
    """Hash of the kernel and host sources under csrc/ without comments, runs
    of whitespace counted as one space: the recorded DRAM traffic stays valid
    across comment-only edits."""
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2607_20739_gb300", "csrc")
    for f in sorted(os.listdir(csrc)):
        if f.endswith((".cu", ".cuh", ".h")):
            with open(os.path.join(csrc, f), encoding="utf-8") as fh:
                h.update(f.encode())
                h.update(" ".join(_strip_comments(fh.read()).split()).encode())
    return h.hexdigest()[:16]


def recorded_traffic(workload: str):
    """DRAM bytes per launch of the dominant kernel from the committed ncu
    summary, if the kernel sources have not changed since it was taken."""
    p = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(p):
        return None
    with open(p) as f:
        d = json.load(f)
    e = d.get(workload)
    if not e or e.get("source_hash") != kernel_source_hash():
        return None
    return e.get("dram_bytes_per_launch")


# ---------------------------------------------------------------------------
# clocks during the timed region
# ---------------------------------------------------------------------------

class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=self.f, stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.f.close()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    rows.append((float(parts[1]), float(parts[2]), parts[5:9]))
                except ValueError:
                    continue
        os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for _, _, r in rows for i, v in enumerate(r) if v.lower() == "active"})
        return {"sm_mhz": statistics.median(r[0] for r in rows), "sm_max_mhz": max(r[1] for r in rows),
                "reasons": reasons, "samples": len(rows)}


# ---------------------------------------------------------------------------
# the fp64 oracle on the host cores (cpu_baseline and --impl reference)
# ---------------------------------------------------------------------------

# workloads whose oracle is also timed on one thread
ONE_THREAD_WORKLOADS = ("fr_n4_logistic_d64", "cr_n8_logistic_d1024")


def cpu_model() -> str:
    """The host CPU's model name (lscpu, else /proc/cpuinfo, else the machine type)."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.lower().startswith("model name"):
                return line.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    try:
        with open("/proc/cpuinfo") as f:
            for line in f:
                if line.lower().startswith("model name"):
                    return line.split(":", 1)[1].strip()
    except OSError:
        pass
    import platform
    return platform.machine()


def time_oracle_one_thread(w: W.Workload, seed: int, mode: str, budget_s: float):
    """time_oracle in a child process whose BLAS and OpenMP pools have one
    thread (the variables take effect only before numpy loads its BLAS).
    Returns (steps/s, sample description) or None."""
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1")
    code = ("import json, bench; from paper_2607_20739_gb300 import workloads as W; "
            f"w = W.WORKLOADS[{w.name!r}]; Xs, ys = W.make_partitions(w, {seed}, threads=1); "
            f"m = W.make_masks(w, 64, {seed + 1000}); "
            f"v, k, el, d = bench.time_oracle(w, Xs, ys, m, {budget_s}, mode={mode!r}); "
            "print(json.dumps([v, d]))")
    try:
        r = subprocess.run([sys.executable, "-c", code], cwd=ROOT, env=env, capture_output=True, text=True,
                           timeout=max(120.0, 20 * budget_s))
    except subprocess.TimeoutExpired:
        return None
    if r.returncode != 0 or not r.stdout.strip():
        return None
    v, d = json.loads(r.stdout.strip().splitlines()[-1])
    return v, d


def time_oracle(w: W.Workload, Xs, ys, masks, budget_s: float, min_steps: int = 2, mode: str = "pgc"):
    """Steady steps/s of the oracle as it stands, and what was timed.

    When the oracle's warm-up and two steady steps fit the budget, whole
    steady steps are timed (warm-up step 0 untimed).  Otherwise a bounded
    sample: the oracle's steady step is n partition gradients (each worker
    evaluates its own) plus the literal decode (a c-slot coded sum per
    received worker); partition gradients are timed one by one for about the
    budget, one coded sum once, and the step time is n t_grad + (n - s) t_coded.
    Returns (steps/s, count, seconds, sample description)."""
    from oracle import pgc_oracle as O
    S = {"FR": O.FR, "CR": O.CR}
    L = {"logistic": O.LOGISTIC, "lsq": O.LSQ, "softmax": O.SOFTMAX}
    Xf = [W.features_as_float(X, w.dtype) for X in Xs]
    gc_cr = mode == "naive_cr" or (mode == "gc" and w.scheme == "CR")
    if mode == "pgc":
        o = O.PGCOracle(S[w.scheme], w.n, w.s, L[w.loss], Xf, ys, w.lr, K=w.K)
    elif gc_cr:
        o = O.NaiveCROracle(w.n, w.s, L[w.loss], Xf, ys, w.lr, draws=W.make_gc_draws(w, GC_DRAWS_SEED), K=w.K,
                            pipelined=mode == "naive_cr")
    else:
        o = {"is_sgd": O.ISSGDOracle, "gc": O.GCFROracle}[mode](w.n, w.s, L[w.loss], Xf, ys, w.lr, K=w.K)
    inner = o if mode == "pgc" or gc_cr else o.inner
    evals_per_step = w.n * (w.c if mode == "gc" else 1)
    t0 = time.perf_counter()
    inner.partition_grad(0)
    t_pg = time.perf_counter() - t0
    if t_pg * (w.n * w.c + 2 * evals_per_step) <= budget_s:
        o.step(masks[0])
        t0 = time.perf_counter()
        k = 0
        while True:
            o.step(masks[(1 + k) % len(masks)])
            k += 1
            el = time.perf_counter() - t0
            if (el >= budget_s and k >= min_steps) or el >= 4 * budget_s:
                break
        return k / el, k, el, f"{k} steady steps of the full {w.name} workload after the warm-up step ({el:.1f} s)"
    # bounded sample
    t0 = time.perf_counter()
    k = 0
    while True:
        inner.partition_grad(k % w.n)
        k += 1
        el = time.perf_counter() - t0
        if (el >= budget_s and k >= 2) or k >= evals_per_step:
            break
    t_grad = el / k
    nslot = 1 if mode == "is_sgd" else w.c                 # gradients per uploaded (coded) gradient
    slots = [inner.partition_grad(j % w.n) if j < 1 else np.ones_like(inner.beta) for j in range(nslot)]
    t1 = time.perf_counter()
    _ = sum(slots[l] for l in range(nslot))
    t_coded = time.perf_counter() - t1
    step_s = evals_per_step * t_grad + (w.n - w.s) * t_coded
    desc = (f"{k} of the {evals_per_step} partition gradients of one steady {w.name} step timed one by one ({el:.1f} s) "
            f"plus one {nslot}-slot coded sum, scaled to (evaluations) t_grad + (n - s) t_coded = {step_s:.2f} s per step")
    return 1.0 / step_s, k, el, desc


# ---------------------------------------------------------------------------
# one GPU only
# ---------------------------------------------------------------------------

SINGLE_GPU_ONLY = ("this path simulates all n workers of a PGC step on one GPU and has no multi-GPU form; "
                   "run bench.py with --gpus 1 (no torchrun)")


def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def refuse_multi_gpu(args) -> None:
    """The GPU arm runs on one GPU: with --gpus > 1, or under a launcher that
    started several ranks, it stops here, before torch or the library is
    imported, so no rank makes a CUDA call."""
    world, _, _ = dist_env()
    if args.gpus != 1 or world != 1:
        print(json.dumps({"error": SINGLE_GPU_ONLY, "gpus": args.gpus, "world_size": world}), file=sys.stderr,
              flush=True)
        raise SystemExit(2)


# ---------------------------------------------------------------------------
# the GPU arm
# ---------------------------------------------------------------------------

def default_steps(w: W.Workload) -> int:
    """Steps of about two seconds of streaming work (20 to 20,000)."""
    per_step_bytes = evaluated_rows(w) * grad_bytes_per_row(w)
    est_s = max(per_step_bytes / 5.0e12, 20e-6)
    if tensor_core_path(w):
        est_s = max(est_s, 4.0 * evaluated_rows(w) * w.d * w.K / 1.2e15)
    return int(min(20000, max(20, 2.0 / est_s)))


def measure(w: W.Workload, K_steps: int, Wu: int, seed: int, mode: str, cpu_seconds, one_thread_seconds,
            torch, dev) -> dict:
    """Every measured field of one workload: device-timed steps/s, the
    per-kernel-group breakdown, the dominant kernel's roofline, the end-to-end
    rate through the public API with host buffers, the clocks during the
    timed region, the simulated wall clock and (cpu_seconds not None) the
    oracle on the host cores."""
    from paper_2607_20739_gb300 import binding as B

    t_gen = time.perf_counter()
    Xs, ys = W.make_partitions(w, seed)
    masks = W.make_masks(w, K_steps + Wu + 1, seed + 1000)
    gen_s = time.perf_counter() - t_gen

    stream = torch.cuda.Stream(device=dev)
    g = B.PGC(w.scheme, w.n, w.s, w.loss, w.dtype, w.d, K=w.K, rows=w.rows(), lr=w.lr, stream=stream, mode=mode)
    g.load(Xs, ys)
    if mode == "naive_cr" or (mode == "gc" and w.scheme == "CR"):
        g.set_gc_encoding(W.make_gc_draws(w, GC_DRAWS_SEED))
    P = w.K * w.d
    gout = torch.empty(P, device=dev)
    wout = torch.empty(P, device=dev)
    step_bytes = evaluated_rows(w) * grad_bytes_per_row(w)
    flush = step_bytes <= L2_BYTES
    flush_buf = torch.empty(256 * 2 ** 20 // 4, device=dev) if flush else None
    mptr = [np.ascontiguousarray(masks[t]) for t in range(len(masks))]

    def do_step(t):
        if flush:
            with torch.cuda.stream(stream):
                flush_buf.zero_()
        g.step(mptr[t], gout, wout, info=False)

    for t in range(Wu):
        do_step(t)
    g.sync()

    # ---- device-timed region: exactly K_steps steps on the library's stream
    # (no per-kernel events: they would break the programmatic-dependent
    # overlap between consecutive step kernels) -----------------------------
    clk = ClockSampler(int(dev.index or 0))
    torch.cuda.synchronize(dev)
    clk.start()
    time.sleep(0.25)
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for t in range(Wu, Wu + K_steps):
        do_step(t)
    ev1.record(stream)
    g.sync()
    torch.cuda.synchronize(dev)
    region_ms = ev0.elapsed_time(ev1)
    clocks = clk.stop()

    # ---- per-kernel-group breakdown: a second pass with events around each
    # group of every step, on the library's stream --------------------------
    k2 = min(K_steps, 2000)
    g.timing(True)
    for t in range(k2):
        do_step(t % len(mptr))
    tim = g.timing_read()
    g.timing(False)
    launches_per_step = sum(tim["launches"]) / max(1, tim["steps"])
    nsteps = max(1, tim["steps"])
    group_ms = [m / nsteps for m in tim["ms"]]
    if flush:
        # the flush between steps is excluded: the step is its kernel groups
        # (groups that launched nothing hold only the events' own time)
        ms_per_step = sum(m for m, nl in zip(group_ms, tim["launches"]) if nl > 0)
    else:
        ms_per_step = region_ms / K_steps
    value = 1000.0 / ms_per_step

    # ---- roofline of the dominant kernel (streaming paths: the gradient
    # kernel, whose launch is the whole step when it carries the fused tail;
    # tensor-core softmax: the slower of the two GEMMs) ----------------------
    peaks, peak_src = load_peaks()
    bound, units, unit, peak = roofline_model(w, peaks)
    single = all(n == 0 for n in tim["launches"][1:]) and tim["launches"][0] == tim["steps"]
    dom = 0
    if tensor_core_path(w) and group_ms[2] > group_ms[0]:
        dom = 2
    grad_ms = ms_per_step if (single and not flush) else group_ms[dom]
    scale = 1e9 if unit == "GB/s" else 1e12
    achieved = units / (grad_ms * 1e-3) / scale
    roofline = {"bound": bound, "achieved": achieved, "peak": peak, "unit": unit, "frac": achieved / peak,
                "peak_source": peak_src, "kernel": kernel_label(w, single, dom), "duration_ms": grad_ms,
                "traffic": recorded_traffic(w.name), "algorithmic_per_launch": units}
    if tensor_core_path(w):
        # the whole step against the burst rate: both contractions' flops
        step_flops = 2.0 * units
        burst = peaks.get("bf16_tflops") or 1900.0
        roofline["step"] = {"flops": step_flops, "achieved": step_flops / (ms_per_step * 1e-3) / 1e12,
                            "peak": burst, "unit": "TFLOP/s",
                            "frac": step_flops / (ms_per_step * 1e-3) / 1e12 / burst,
                            "note": "logits X W^T and gradient R^T X, 2 rows d K flops each, over the whole "
                                    "step (both GEMMs, the commit into the stores and the decode) against the "
                                    "burst bf16 rate"}

    # ---- end to end through the public API with host buffers -------------
    gh = torch.empty(P, dtype=torch.float32).pin_memory()
    wh = torch.empty(P, dtype=torch.float32).pin_memory()
    e2e_steps = max(10, min(K_steps, 2000))
    t0 = time.perf_counter()
    for t in range(e2e_steps):
        g.step(mptr[t % len(mptr)], gh, wh, info=False)
    e2e_s = time.perf_counter() - t0
    e2e_value = e2e_steps / e2e_s

    # ---- the GC-CR modes' decoding coefficients alpha_{m,k} (§V-A): their
    # range, read after each of some untimed steps ------------------------
    alpha = None
    if mode == "naive_cr" or (mode == "gc" and w.scheme == "CR"):
        amax, amin, big = -float("inf"), float("inf"), 0
        na = min(200, len(mptr))
        for t in range(na):
            g.step(mptr[t], None, None, info=False)
            _, (hi, lo) = g.gc_decode()
            amax, amin = max(amax, hi), min(amin, lo)
            big += int(max(abs(hi), abs(lo)) > 100.0)
        alpha = {"max": amax, "min": amin, "steps": na, "steps_with_abs_over_100": big,
                 "note": "alpha_{m,k} = d_m(J) c_{j_m,l} derived on the device each step (untimed steps)"}
    g.close()
    del gout, wout, flush_buf, gh, wh
    torch.cuda.empty_cache()

    # ---- cpu baseline: the oracle as it stands, on the host cores ---------
    cpu = None
    if cpu_seconds is not None:
        v, k, el, desc = time_oracle(w, Xs, ys, masks, cpu_seconds, mode=mode)
        cpu = {"value": v, "unit": "steps/s", "cores": os.cpu_count(), "kind": "oracle",
               "sample": desc + "; fp64 numpy, BLAS threads = all cores", "cpu_model": cpu_model()}
        if w.name in ONE_THREAD_WORKLOADS and one_thread_seconds:
            one = time_oracle_one_thread(w, seed, mode, one_thread_seconds)
            if one is not None:
                cpu["value_1thread"] = one[0]
                cpu["sample_1thread"] = one[1] + "; fp64 numpy, one thread"
    del Xs, ys

    # ---- simulated wall clock of a step (the paper's time per step, PGC vs
    # DGD / IS-SGD / GC): the device-timed step less the decode is the
    # workers' compute, the decode is the master's; seeded delays in units of
    # the compute time ------------------------------------------------------
    from paper_2607_20739_gb300 import wallclock as WC
    # (paths whose gradient kernel decodes in its own tail launch no decode
    # kernel: their decode group holds only the events' own time)
    decode_ms = min(group_ms[4], ms_per_step) if tim["launches"][4] > 0 else 0.0
    compute_ms = ms_per_step - decode_ms
    # one partition per worker: a GC run evaluates c partitions per worker
    compute_s = compute_ms * 1e-3 / (w.c if mode == "gc" else 1)
    delays = W.draw_delays(w, K_steps + Wu + 1, seed + 1000)[Wu:Wu + K_steps]
    sim = WC.summary(delays, w.n, w.s, compute_s, compute_s, decode_ms * 1e-3)
    sim["model"] = ("each worker finishes after (partitions evaluated) x compute + delay; the master waits for "
                    "the n - s fastest (pgc, is_sgd, gc with c partitions per worker) or all n (dgd), then decodes; "
                    "compute = the device-timed step less its decode kernel (per partition), decode = the decode "
                    "kernel's event time; delays are the seeded draws that pick the stragglers, in units of the "
                    "compute time")

    uniq = evaluated_rows(w)
    out = {
        "value": value, "unit": "steps/s", "steps": K_steps, "warmup": Wu, "ms_per_step": ms_per_step,
        "dtype": "f32" if w.dtype == "f32" else "bf16-in/f32-acc",
        "config": {"workload": w.name, "scheme": w.scheme, "n": w.n, "s": w.s, "loss": w.loss, "d": w.d, "K": w.K,
                   "rows_per_partition": w.m, "features": w.dtype, "parallelism": "single GPU", "mode": mode,
                   "l2": ("flushed between steps (256 MiB write, excluded from step time)" if flush else
                          f"inputs larger than L2: {step_bytes / 2**20:.0f} MiB streamed per step")},
        "samples_per_s_unique": value * uniq,
        "samples_per_s_worker": value * sum(w.rows()),
        "kernel_ms_per_step": {B.KERNEL_GROUPS[i]: group_ms[i] for i in range(len(B.KERNEL_GROUPS))
                               if tim["launches"][i] > 0},
        "kernel_timing_note": "per-group CUDA events from a separate pass; events between launches "
                              "serialise the dependent-launch overlap, so these sum to more than ms_per_step",
        "roofline": roofline,
        "cpu_baseline": cpu,
        "e2e": {"value": e2e_value, "unit": "steps/s", "steps": e2e_steps, "h2d_bytes_per_step": w.n,
                "d2h_bytes_per_step": 2 * P * 4},
        "gpu_launches": int(round(launches_per_step * K_steps)),
        "simulated_wall_clock": sim,
        "clocks": clocks,
        "input_generation_s": gen_s,
    }
    if alpha is not None:
        out["decoding_coefficients"] = alpha
    return out


def run_ours(args):
    refuse_multi_gpu(args)
    import torch
    if not torch.cuda.is_available():
        raise SystemExit("bench.py: no CUDA device (the GPU arm has no CPU fallback)")
    torch.cuda.set_device(0)
    dev = torch.device("cuda", 0)

    head = workload_from_args(args)
    K_steps = args.steps or default_steps(head)
    Wu = max(3, args.warmup)
    cpu_s = None if args.no_cpu_baseline else args.cpu_seconds
    res = measure(head, K_steps, Wu, args.seed, args.mode, cpu_s, min(8.0, args.cpu_seconds), torch, dev)

    per = None
    if args.workload is None and not args.no_per_workload:
        # every other workload in the same invocation, each over its own
        # step count (about two seconds of work) with 5 warm-up steps
        per = {}
        cpu_o = None if args.no_cpu_baseline else min(args.cpu_seconds, 8.0)
        for name in W.WORKLOAD_ORDER:
            if name == head.name:
                continue
            w = W.WORKLOADS[name]
            per[name] = measure(w, default_steps(w), 5, args.seed, args.mode, cpu_o, min(5.0, args.cpu_seconds),
                                torch, dev)

    line = {
        "metric": METRIC, "value": res["value"], "unit": "steps/s", "n_gpus": 1, "steps": K_steps, "warmup": Wu,
        "ms_per_step": res["ms_per_step"], "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": res["dtype"],
        "data": f"synthetic, seeded (seed {args.seed}); {head.features} features, planted-model labels, "
                f"{head.delays} straggler delays",
    }
    for k, v in res.items():
        if k not in line:
            line[k] = v
    if per is not None:
        line["per_workload"] = per
        line["per_workload_note"] = ("the other workloads, measured in this invocation after the headline, each "
                                     "over its own step count (about two seconds of device work) after 5 warm-up "
                                     "steps; every field as at the top level")
    print(json.dumps(line), flush=True)


def run_reference(args):
    """The fp64 oracle on the host cores (CPU only: no CUDA call).  Under a
    launcher that started several ranks only rank 0 runs it."""
    world, rank, _ = dist_env()
    if rank != 0:
        return
    w = workload_from_args(args)
    K_steps = args.steps or 3
    Xs, ys = W.make_partitions(w, args.seed)
    masks = W.make_masks(w, K_steps + max(3, args.warmup) + 1, args.seed + 1000)
    budget = min(args.cpu_seconds, 60.0)
    v, k, el, desc = time_oracle(w, Xs, ys, masks, budget, min_steps=min(K_steps, 3), mode=args.mode)
    if "steady steps" not in desc:
        k = max(1, int(round(el * v)))         # sampled: whole-step equivalents of the timed work
    line = {
        "impl": "reference", "metric": METRIC, "value": v, "unit": "steps/s", "n_gpus": world, "steps": k,
        "warmup": 1, "ms_per_step": 1000.0 / v, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "f64", "data": f"synthetic, seeded (seed {args.seed})",
        "config": {"workload": w.name, "scheme": w.scheme, "n": w.n, "s": w.s, "loss": w.loss, "d": w.d, "K": w.K,
                   "rows_per_partition": w.m, "mode": args.mode},
        "cpu_baseline": {"value": v, "unit": "steps/s", "cores": os.cpu_count(), "kind": "oracle",
                         "sample": desc, "cpu_model": cpu_model()},
        "e2e": {"value": v, "unit": "steps/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def main(argv=None):
    args = parse_args(argv)
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
