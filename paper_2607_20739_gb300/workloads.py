"""Seeded synthetic workloads for the PGC hot path.

This module only draws inputs: partition features and labels, and per-step
straggler masks.  It holds none of the method's arithmetic (no placement, no
gradients, no encoding or decoding), so both the CUDA path and the fp64 oracle
can take their inputs from it.

Workloads (one per row; each stands in for a dataset the paper trains on):

  fr_n4_logistic_d64     FR n=4  s=1  logistic   d=64    m=256  fp32 N(0,1)
  cr_n8_logistic_d1024   CR n=8  s=2  logistic   d=1024  m=8192 fp32 N(0,1)
  fr_n32_softmax_k10     FR n=32 s=3  softmax K=10   d=3072 m=4096 bf16 U[0,1)
                         (image-like, shaped like CIFAR-10's 32x32x3 inputs)
  cr_n64_lsq_d16384      CR n=64 s=4  least squares d=16384 m=2048 fp32 N(0,1)
  cr_n128_softmax_k1000  CR n=128 s=7 softmax K=1000 d=4096 m=1024 bf16 N(0,1)
                         (shaped like the downsampled-ImageNet runs of §VI-B)

Labels come from a planted model: w* ~ N(0, I/d) (rows of W* likewise).
Logistic: y ~ Bernoulli(sigmoid(x.w*)).  Least squares: y = x.w* + N(0, 0.1^2).
Softmax: y = argmax_k (W* x + Gumbel noise)_k, i.e. a draw from softmax(W* x).

Straggler masks: per step each worker draws a delay; the s slowest are the
stragglers (ties: the lower worker index counts as faster).  Delay models:
uniform (one uniform straggler), shifted exponential (shift 1, rate 1, the
exponential delays of §VI-B shifted by a unit compute time) and Pareto(2).

Every array is a deterministic function of (workload, seed, partition or
step): partition k uses the generator ``default_rng([seed, 1, k])``, the
planted model ``default_rng([seed, 0])`` and the delays
``default_rng([seed, 2])``.
"""

from __future__ import annotations

import concurrent.futures as _cf
import dataclasses
import os

import numpy as np


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    scheme: str            # "FR" or "CR"
    n: int                 # workers = partitions
    s: int                 # stragglers tolerated; c = s + 1
    loss: str              # "logistic", "lsq" or "softmax"
    dtype: str             # "f32" or "bf16" (feature storage)
    d: int                 # features per sample
    K: int                 # classes (1 unless softmax)
    m: int | tuple         # rows per partition (int, or one per partition)
    lr: float
    T: int                 # steps of the run
    features: str          # "normal" or "uniform"
    delays: str            # "uniform", "shifted_exp" or "pareto2"

    @property
    def c(self) -> int:
        return self.s + 1

    def rows(self) -> list[int]:
        if isinstance(self.m, int):
            return [self.m] * self.n
        return list(self.m)

    def replace(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


# The five workloads measured and checked.  Learning rates other than the first
# are not given anywhere; these keep the fp64 loss decreasing on every one.
WORKLOADS = {
    "fr_n4_logistic_d64": Workload(
        "fr_n4_logistic_d64", "FR", 4, 1, "logistic", "f32", 64, 1, 256,
        0.1, 20, "normal", "uniform"),
    "cr_n8_logistic_d1024": Workload(
        "cr_n8_logistic_d1024", "CR", 8, 2, "logistic", "f32", 1024, 1, 8192,
        0.1, 200, "normal", "shifted_exp"),
    "fr_n32_softmax_k10": Workload(
        "fr_n32_softmax_k10", "FR", 32, 3, "softmax", "bf16", 3072, 10, 4096,
        1e-3, 500, "uniform", "shifted_exp"),
    "cr_n64_lsq_d16384": Workload(
        "cr_n64_lsq_d16384", "CR", 64, 4, "lsq", "f32", 16384, 1, 2048,
        0.05, 300, "normal", "pareto2"),
    "cr_n128_softmax_k1000": Workload(
        "cr_n128_softmax_k1000", "CR", 128, 7, "softmax", "bf16", 4096, 1000, 1024,
        0.1, 200, "normal", "shifted_exp"),
}

WORKLOAD_ORDER = list(WORKLOADS)


# ----------------------------------------------------------------------------
# bf16 storage (features are rounded to bf16 once, at generation)
# ----------------------------------------------------------------------------

def f32_to_bf16_bits(a: np.ndarray) -> np.ndarray:
    """Round float32 values to bf16 (nearest, ties to even); returns uint16 bits."""
    u = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32)
    bias = ((u >> np.uint32(16)) & np.uint32(1)) + np.uint32(0x7FFF)
    return ((u + bias) >> np.uint32(16)).astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bits (uint16) to float32."""
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def features_as_float(X: np.ndarray, dtype: str) -> np.ndarray:
    """The exact values a feature array stands for, as float32."""
    return bf16_bits_to_f32(X) if dtype == "bf16" else np.asarray(X, dtype=np.float32)


# ----------------------------------------------------------------------------
# Partitions
# ----------------------------------------------------------------------------

def planted_model(w: Workload, seed: int) -> np.ndarray:
    """w* (shape [d]) or W* (shape [K, d]) with entries N(0, 1/d)."""
    rng = np.random.default_rng([seed, 0])
    shape = (w.K, w.d) if w.loss == "softmax" else (w.d,)
    return rng.standard_normal(shape) / np.sqrt(w.d)


def make_partition(w: Workload, seed: int, k: int, planted: np.ndarray | None = None):
    """Features X_k ([m_k, d]; float32, or uint16 bf16 bits) and labels y_k of D_k."""
    if planted is None:
        planted = planted_model(w, seed)
    m = w.rows()[k]
    rng = np.random.default_rng([seed, 1, k])
    if w.features == "normal":
        Xf = rng.standard_normal((m, w.d), dtype=np.float32)
    elif w.features == "uniform":
        Xf = rng.random((m, w.d), dtype=np.float32)
    else:
        raise ValueError(w.features)
    if w.dtype == "bf16":
        X = f32_to_bf16_bits(Xf)
        Xv = bf16_bits_to_f32(X)
    elif w.dtype == "f32":
        X = Xf
        Xv = Xf
    else:
        raise ValueError(w.dtype)
    if w.loss == "logistic":
        z = Xv.astype(np.float64) @ planted
        p = 1.0 / (1.0 + np.exp(-z))
        y = (rng.random(m) < p).astype(np.float32)
    elif w.loss == "lsq":
        z = Xv.astype(np.float64) @ planted
        y = (z + 0.1 * rng.standard_normal(m)).astype(np.float32)
    elif w.loss == "softmax":
        Z = Xv @ planted.T.astype(np.float32)
        g = rng.gumbel(size=Z.shape).astype(np.float32)
        y = np.argmax(Z + g, axis=1).astype(np.int32)
    else:
        raise ValueError(w.loss)
    return X, y


def make_partitions(w: Workload, seed: int, threads: int | None = None):
    """All n partitions (lists Xs, ys), generated in parallel threads."""
    planted = planted_model(w, seed)
    threads = threads or min(w.n, os.cpu_count() or 1)
    if threads <= 1 or w.n == 1:
        parts = [make_partition(w, seed, k, planted) for k in range(w.n)]
    else:
        with _cf.ThreadPoolExecutor(threads) as ex:
            parts = list(ex.map(lambda k: make_partition(w, seed, k, planted), range(w.n)))
    return [p[0] for p in parts], [p[1] for p in parts]


# ----------------------------------------------------------------------------
# Straggler masks
# ----------------------------------------------------------------------------

def draw_delays(w: Workload, steps: int, seed: int) -> np.ndarray:
    """Per-step, per-worker simulated delays, shape [steps, n] (float64)."""
    rng = np.random.default_rng([seed, 2])
    u = rng.random((steps, w.n))
    if w.delays == "uniform":
        return u
    if w.delays == "shifted_exp":
        return 1.0 - np.log1p(-u)              # 1 + Exp(rate 1)
    if w.delays == "pareto2":
        return (1.0 - u) ** (-0.5)             # Pareto, x_m = 1, alpha = 2
    raise ValueError(w.delays)


def make_gc_draws(w: Workload, seed: int) -> np.ndarray:
    """float64 [s, n-1] standard normal draws: the random numbers of GC-CR's
    cyclic-repetition encoding (§V-A), passed to both sides as an input."""
    return np.random.default_rng(seed).standard_normal((w.s, w.n - 1))


def make_masks(w: Workload, steps: int, seed: int) -> np.ndarray:
    """uint8 [steps, n]; 1 marks the s workers with the largest delay that step."""
    D = draw_delays(w, steps, seed)
    masks = np.zeros((steps, w.n), dtype=np.uint8)
    if w.s == 0:
        return masks
    idx = np.arange(w.n)
    for t in range(steps):
        order = np.lexsort((idx, D[t]))       # by delay, then by index (lower = faster)
        masks[t, order[w.n - w.s:]] = 1
    return masks
