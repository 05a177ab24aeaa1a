"""Simulated wall clock of one training step (§VI, "time per step").

Each worker finishes a step after its compute time plus a seeded random
delay.  The master decodes once it holds what the scheme needs:

    scheme   partitions evaluated per worker   workers the master waits for
    pgc      1                                  n - s  (§IV, §V)
    is_sgd   1                                  n - s
    gc       c = s + 1                          n - s
    dgd      1                                  n      (c = 1, s = 0)

so the step takes the (waited-for)-th smallest of (partitions x t_compute +
delay_i) plus the master's decode.  The compute time of one partition per
worker is the measured GPU time of the step's gradient evaluation (all
workers evaluate concurrently), the delays are the workload's seeded draws
(the ones that pick the stragglers) in units of `delay_unit_s`, and the
decode time is the measured decode.  IS-GC is not modelled (its code is only
cited by the paper).
"""

from __future__ import annotations

import numpy as np

SCHEMES = ("pgc", "is_sgd", "gc", "dgd")


def partitions_per_worker(scheme: str, c: int) -> int:
    return c if scheme == "gc" else 1


def waited_for(scheme: str, n: int, s: int) -> int:
    return n if scheme == "dgd" else n - s


def step_times(delays, n: int, s: int, compute_s: float, delay_unit_s: float, decode_s: float = 0.0) -> dict:
    """Per-step simulated times (seconds) of every scheme; delays [steps, n]."""
    D = np.asarray(delays, dtype=np.float64)
    if D.ndim != 2 or D.shape[1] != n:
        raise ValueError("delays must have shape [steps, n]")
    if not 0 <= s < n:
        raise ValueError("need 0 <= s < n")
    c = s + 1
    out = {}
    for sch in SCHEMES:
        finish = partitions_per_worker(sch, c) * compute_s + delay_unit_s * D
        kth = np.sort(finish, axis=1)[:, waited_for(sch, n, s) - 1]
        out[sch] = kth + decode_s
    return out


def summary(delays, n: int, s: int, compute_s: float, delay_unit_s: float, decode_s: float = 0.0) -> dict:
    """Mean per-step time (us) of each scheme and its ratio to DGD."""
    t = step_times(delays, n, s, compute_s, delay_unit_s, decode_s)
    mean = {k: float(np.mean(v)) for k, v in t.items()}
    return {
        "per_step_us": {k: v * 1e6 for k, v in mean.items()},
        "normalized_to_dgd": {k: v / mean["dgd"] for k, v in mean.items()},
        "compute_us": compute_s * 1e6,
        "delay_unit_us": delay_unit_s * 1e6,
        "decode_us": decode_s * 1e6,
        "steps": int(np.asarray(delays).shape[0]),
    }
