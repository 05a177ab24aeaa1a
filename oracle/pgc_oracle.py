"""Plain, slow fp64 CPU oracle of Pipelined Gradient Coding (PGC).

TEST INFRASTRUCTURE ONLY.  Nothing in the product path (the CUDA library and
its Python binding) imports, calls or links this module; only the tests,
``__graft_entry__.smoke()`` and the ``cpu_baseline`` / ``--impl reference``
legs of ``bench.py`` do.  It shares no code, tables or constants with the GPU
path.  It receives its inputs as plain arrays (from the seeded workload
generators) and never reads anything the GPU produced, except where a test
feeds it the GPU's parameters on purpose ("teacher forcing").

What it computes, step by step, in fp64, literally per worker (no sharing of
work between workers that hold the same partitions):

* §III    dataset placement for fractional repetition (FR) and cyclic
          repetition (CR); the ERM objective F and the SGD update.
* §IV-A   PGC-FR: worker W_i evaluates one partition per step, rotating
          through its c partitions, keeps the latest gradient of each, uploads
          their sum; the master takes one coded gradient per group and scales
          the sum by 1/n.  Step t = 0 is the warm-up in which every worker
          evaluates all c of its partitions at beta^(0).
* §V-B    PGC-CR: same rotation on the cyclic placement; every coefficient is
          1; the master sums the n - s received coded gradients and scales by
          1/(n mu) = 1/((n - s) c).
* §VI-A   stragglers still evaluate and store their gradients; they are only
          left out of the decode.

Readings where the paper is silent (each is also listed in the design notes):
  R1  a partition gradient g_k is the MEAN of the per-sample gradients over
      D_k, so FR with equal partition sizes and no staleness is exactly the
      full-data gradient, as DGD's (1/n) sum_i g_i in §III implies;
  R2  t = 0 decodes and updates like every other step and is the first step;
  R3  CR at t = 0 decodes with the PGC-CR rule on an all-current store;
  R5  an FR group is represented by its lowest-index non-straggler;
  R6  a straggler mask has exactly s ones;
  R7  losses: logistic cross-entropy with y in {0, 1}; least squares
      (1/2)(x.beta - y)^2; softmax cross-entropy; no bias, no regulariser.

Baselines (§VI-A), for comparison on the same kernels: IS-SGD (the master
averages the n - s fastest workers' own-partition gradients) and GC with FR
placement (every worker evaluates its c partitions every step).

§V-A, the naive pipelined construction on cyclic repetition: PGC-CR's
schedule and placement, but each worker uploads GC-CR's weighted sum
sum_l c_{j,l} * (its latest copy of g_{(j+l) mod n}) and the master applies
GC-CR's straggler-dependent decode weights d_m(J); alpha_{m,k} = d_m c_{j_m,l}
are the decoding coefficients whose range §V-A tracks.  The coefficients
c_{j,l} are those of the cyclic-repetition construction of gradient coding,
which §V-A cites (Tandon et al., ICML 2017) without restating; it is
restated below from its definition.  With every copy current (GC-CR proper:
all c partitions evaluated each step) the decode is exact.  Further readings:
  R14 the naive and GC-CR decodes are scaled by 1/n, like FR's, so that with
      current copies they equal DGD's (1/n) sum_k g_k;
  R15 the construction's random matrix arrives as draws [s][n-1]; its last
      column is minus the row sums (so H 1 = 0);
  R16 the range of alpha is taken over the pairs the definition names:
      received workers j_m and the c partitions each holds.

Parity of whole trajectories is pinned only through the invariants the paper
proves (eq. cr-fullsum, eq. cr-unbiased, the FR / GC equivalence and the DGD
special case); there is no printed trajectory to compare with.
"""

from __future__ import annotations

import itertools
import math

import numpy as np

FR = 0
CR = 1
LOGISTIC = 0
LSQ = 1
SOFTMAX = 2

SCHEME_NAMES = {FR: "FR", CR: "CR"}
LOSS_NAMES = {LOGISTIC: "logistic", LSQ: "lsq", SOFTMAX: "softmax"}


# ----------------------------------------------------------------------------
# Placement and schedule (§III, §IV-A, §V-B)
# ----------------------------------------------------------------------------

def holdings(scheme: int, n: int, c: int) -> list[list[int]]:
    """Partitions held by each worker, indexed [worker][slot l], l = 0..c-1.

    FR (§III, §IV-A): needs c | n; W_i holds D_{jc}, ..., D_{jc+c-1} with
    j = floor(i / c), so slot l holds D_{jc+l}.
    CR (§III, §V-B): W_i holds D_{(i+l) mod n} for l = 0..c-1.
    """
    if n < 1 or c < 1 or c > n:
        raise ValueError(f"need 1 <= c <= n, got n={n} c={c}")
    if scheme == FR:
        if n % c != 0:
            raise ValueError(f"FR needs c | n, got n={n} c={c}")
        return [[(i // c) * c + l for l in range(c)] for i in range(n)]
    if scheme == CR:
        return [[(i + l) % n for l in range(c)] for i in range(n)]
    raise ValueError(f"unknown scheme {scheme}")


def fr_group(i: int, c: int) -> int:
    """Group j = floor(i / c) of FR worker W_i (§IV-A)."""
    return i // c


def evaluated_slot(t: int, c: int) -> int | None:
    """Slot a worker evaluates at step t >= 1: (t - 1) mod c (§IV-A, §V-B).

    None at the warm-up step t = 0, where all c slots are evaluated (§IV-A).
    """
    if t == 0:
        return None
    return (t - 1) % c


def evaluated_partition(scheme: int, n: int, c: int, i: int, t: int) -> int | None:
    """Partition W_i evaluates at step t >= 1.

    FR: D_{jc + ((t-1) mod c)} (§IV-A).  CR: D_{(i + ((t-1) mod c)) mod n} (§V-B).
    Both are the partition in slot (t-1) mod c of the worker's holdings.
    """
    l = evaluated_slot(t, c)
    if l is None:
        return None
    if scheme == FR:
        return fr_group(i, c) * c + l
    return (i + l) % n


# ----------------------------------------------------------------------------
# Loss and per-partition gradient (§III: F = (1/d) sum f, g_i on D_i)
# ----------------------------------------------------------------------------

def _as64(a) -> np.ndarray:
    return np.asarray(a, dtype=np.float64)


def sample_losses(loss: int, X, y, beta) -> np.ndarray:
    """Per-sample loss f(beta; x, y) for every row x of X (reading R7).

    logistic: log(1 + exp(x.beta)) - y x.beta
    lsq:      (1/2) (x.beta - y)^2
    softmax:  log sum_k exp(w_k.x) - w_y.x,  beta = W with rows w_k
    """
    X = _as64(X)
    beta = _as64(beta)
    if loss == LOGISTIC:
        z = X @ beta.reshape(-1)
        return np.logaddexp(0.0, z) - _as64(y) * z
    if loss == LSQ:
        z = X @ beta.reshape(-1)
        return 0.5 * (z - _as64(y)) ** 2
    if loss == SOFTMAX:
        Z = X @ beta.T                                   # [m, K] logits
        zmax = Z.max(axis=1, keepdims=True)
        lse = zmax[:, 0] + np.log(np.exp(Z - zmax).sum(axis=1))
        yi = np.asarray(y, dtype=np.int64)
        return lse - Z[np.arange(Z.shape[0]), yi]
    raise ValueError(f"unknown loss {loss}")


def partition_gradient(loss: int, X, y, beta) -> np.ndarray:
    """g_k = (1/m_k) sum over the rows of D_k of grad f (reading R1), fp64.

    logistic: (1/m) X^T (sigma(X beta) - y)
    lsq:      (1/m) X^T (X beta - y)
    softmax:  (1/m) (softmax(X W^T) - onehot(y))^T X, shape [K, d]
    """
    X = _as64(X)
    beta = _as64(beta)
    m = X.shape[0]
    if loss == LOGISTIC:
        z = X @ beta.reshape(-1)
        r = 1.0 / (1.0 + np.exp(-z)) - _as64(y)
        return (X.T @ r) / m
    if loss == LSQ:
        r = X @ beta.reshape(-1) - _as64(y)
        return (X.T @ r) / m
    if loss == SOFTMAX:
        Z = X @ beta.T
        Z = Z - Z.max(axis=1, keepdims=True)
        P = np.exp(Z)
        P /= P.sum(axis=1, keepdims=True)
        yi = np.asarray(y, dtype=np.int64)
        P[np.arange(m), yi] -= 1.0
        return (P.T @ X) / m
    raise ValueError(f"unknown loss {loss}")


def full_loss(loss: int, Xs, ys, beta) -> float:
    """F(beta) = (1/sum_k m_k) sum over every sample of f (§III)."""
    tot = 0.0
    cnt = 0
    for X, y in zip(Xs, ys):
        tot += float(sample_losses(loss, X, y, beta).sum())
        cnt += len(y)
    return tot / cnt


# ----------------------------------------------------------------------------
# Decode rules (§IV-A, §V-B)
# ----------------------------------------------------------------------------

def received_set(mask) -> list[int]:
    """Workers whose coded gradient reaches the master: mask[i] == 0."""
    return [i for i, b in enumerate(mask) if int(b) == 0]


def check_mask(mask, n: int, s: int) -> None:
    """A mask marks exactly s stragglers with 1 and the rest with 0 (reading R6)."""
    if len(mask) != n:
        raise ValueError("mask length != n")
    vals = [int(b) for b in mask]
    if any(v not in (0, 1) for v in vals) or sum(vals) != s:
        raise ValueError("mask must hold exactly s ones and n - s zeros")


def fr_representatives(mask, n: int, c: int) -> list[int]:
    """Lowest-index non-straggler of each FR group (reading R5, §IV-A)."""
    reps = []
    for j in range(n // c):
        alive = [i for i in range(j * c, (j + 1) * c) if int(mask[i]) == 0]
        if not alive:
            raise ValueError(f"FR group {j} has no non-straggler")
        reps.append(alive[0])
    return reps


def decode_coefficients(scheme: int, n: int, s: int, mask) -> np.ndarray:
    """Weight a_i the master gives worker W_i's coded gradient.

    FR (§IV-A, §IV-B): one coded gradient per group, summed, times 1/n, so
    a_i = 1/n for each group's representative and 0 for everyone else.
    CR (§V-B): a_i = 1/(n mu) = 1/((n - s) c) for every received worker.
    """
    c = s + 1
    a = np.zeros(n, dtype=np.float64)
    if scheme == FR:
        for r in fr_representatives(mask, n, c):
            a[r] = 1.0 / n
    else:
        mu = (n - s) * c / n
        for i in received_set(mask):
            a[i] = 1.0 / (n * mu)
    return a


def appearance_counts(scheme: int, n: int, s: int, mask) -> np.ndarray:
    """|N_k|: how often partition k appears among the received workers' holdings (§V-B)."""
    c = s + 1
    hold = holdings(scheme, n, c)
    N = np.zeros(n, dtype=np.int64)
    for i in received_set(mask):
        for k in hold[i]:
            N[k] += 1
    return N


# ----------------------------------------------------------------------------
# GC-CR encoding and decoding coefficients (§V-A)
# ----------------------------------------------------------------------------

def gc_cr_encoding(n: int, s: int, draws=None) -> np.ndarray:
    """Encoding matrix B [n][n] of gradient coding with cyclic repetition.

    The construction §V-A cites (Tandon et al. 2017, cyclic repetition):
    H = [draws | -(row sums of draws)] is s x n, so H 1 = 0.  Row j of B is
    supported on {j, j+1, ..., j+s} mod n, has B[j][j] = 1, and its other s
    entries x solve H[:, {j+1..j+s}] x = -H[:, j]; then H B[j]^T = 0.  So the
    rows of B and the all-ones vector all lie in the null space of H, which
    has dimension n - s for generic draws, and any n - s rows of B span it:
    the master can always find d with sum_m d_m B[j_m] = 1.
    Worker j's encoding coefficient c_{j,l} is B[j][(j + l) mod n].
    """
    B = np.zeros((n, n), dtype=np.float64)
    if s == 0:
        np.fill_diagonal(B, 1.0)
        return B
    D = _as64(draws).reshape(s, n - 1)
    H = np.concatenate([D, -D.sum(axis=1, keepdims=True)], axis=1)
    for j in range(n):
        rest = [(j + l) % n for l in range(1, s + 1)]
        B[j, j] = 1.0
        B[j, rest] = np.linalg.solve(H[:, rest], -H[:, j])
    return B


def encoding_coefficients(B: np.ndarray, c: int) -> np.ndarray:
    """c_{j,l} = B[j][(j + l) mod n] for l = 0..c-1 (§V-A), shape [n][c]."""
    n = B.shape[0]
    return np.array([[B[j, (j + l) % n] for l in range(c)] for j in range(n)])


def gc_decode_weights(B: np.ndarray, mask) -> np.ndarray:
    """GC-CR's decode weights d(J) (§V-A): sum_{m} d_m B[j_m] = 1 over the
    received workers J; d is 0 for stragglers.  Raises if no such d exists."""
    n = B.shape[0]
    J = received_set(mask)
    A = B[J, :].T                                      # n equations, |J| unknowns
    sol, _, rank, _ = np.linalg.lstsq(A, np.ones(n), rcond=None)
    scale = 1.0 + np.abs(sol).max() * np.abs(A).max() if len(J) else 1.0
    if rank < len(J) or np.abs(A @ sol - 1.0).max() > 1e-8 * scale:
        raise ValueError("this encoding cannot decode the straggler pattern")
    d = np.zeros(n)
    d[J] = sol
    return d


def decoding_alpha(B: np.ndarray, d: np.ndarray, mask, c: int) -> dict:
    """alpha_{m,k} = d_m c_{j_m,l} with (j_m + l) mod n = k (§V-A), keyed
    (j_m, k), for every received worker j_m and each partition it holds."""
    n = B.shape[0]
    return {(j, (j + l) % n): d[j] * B[j, (j + l) % n] for j in received_set(mask) for l in range(c)}


# ----------------------------------------------------------------------------
# The PGC training loop, literally per worker (§IV-A, §V-B, §VI-A)
# ----------------------------------------------------------------------------

class PGCOracle:
    """One simulated PGC run: n workers, s stragglers, c = s + 1.

    Xs[k], ys[k] are partition D_k's rows and labels.  beta has shape [d]
    (logistic, lsq) or [K, d] (softmax).  Each worker keeps its own store
    ``ring[i][l]`` of the latest gradient evaluated for the partition in its
    slot l, with ``ring_step[i][l]`` = the step it was evaluated at (the
    s(t, i) / s(t, i, j) bookkeeping of §IV-B and §V-B).
    """

    def __init__(self, scheme, n, s, loss, Xs, ys, lr, beta0=None, K=1):
        if s < 0 or n < 1:
            raise ValueError("need n >= 1 and s >= 0")
        self.scheme = scheme
        self.n = n
        self.s = s
        self.c = s + 1
        self.loss = loss
        self.Xs = list(Xs)
        self.ys = list(ys)
        if len(self.Xs) != n or len(self.ys) != n:
            raise ValueError("need one partition per worker (n partitions)")
        self.lr = float(lr)
        self.d = int(np.asarray(self.Xs[0]).shape[1])
        self.K = int(K)
        shape = (self.K, self.d) if loss == SOFTMAX else (self.d,)
        self.beta = np.zeros(shape) if beta0 is None else _as64(beta0).reshape(shape).copy()
        self.hold = holdings(scheme, n, self.c)
        self.t = 0
        self.ring = [[None] * self.c for _ in range(n)]
        self.ring_step = [[None] * self.c for _ in range(n)]
        self.grad_evals = 0

    # -- pieces -----------------------------------------------------------
    def partition_grad(self, k, beta=None):
        """Gradient of partition D_k at beta (default: current beta^(t))."""
        self.grad_evals += 1
        b = self.beta if beta is None else beta
        return partition_gradient(self.loss, self.Xs[k], self.ys[k], b)

    def coded(self, i):
        """Coded gradient of W_i: the all-ones sum of its c stored gradients
        (§IV-A: sum_l g^{(t-l)}_{jc+((t-1-l) mod c)}; §V-B likewise)."""
        return sum(self.ring[i][l] for l in range(self.c))

    def evaluate(self):
        """Every worker, stragglers included (§V-B, §VI-A), evaluates at beta^(t)."""
        t = self.t
        if t == 0:
            for i in range(self.n):
                for l in range(self.c):
                    self.ring[i][l] = self.partition_grad(self.hold[i][l])
                    self.ring_step[i][l] = 0
            return
        l = evaluated_slot(t, self.c)
        for i in range(self.n):
            self.ring[i][l] = self.partition_grad(self.hold[i][l])
            self.ring_step[i][l] = t

    def decode(self, mask):
        """Master's aggregate sum_i a_i * coded_i (§IV-A, §V-B)."""
        a = decode_coefficients(self.scheme, self.n, self.s, mask)
        g = np.zeros_like(self.beta)
        for i in range(self.n):
            if a[i] != 0.0:
                g = g + a[i] * self.coded(i)
        return g

    def loss_value(self):
        return full_loss(self.loss, self.Xs, self.ys, self.beta)

    # -- one training step --------------------------------------------------
    def step(self, mask):
        """Take step t: evaluate, encode, decode with the received set, update."""
        check_mask(mask, self.n, self.s)
        t = self.t
        self.evaluate()
        g = self.decode(mask)
        rec = {
            "t": t,
            "slot": -1 if t == 0 else evaluated_slot(t, self.c),
            "eval_partition": [-1 if t == 0 else evaluated_partition(self.scheme, self.n, self.c, i, t)
                               for i in range(self.n)],
            "fr_rep": fr_representatives(mask, self.n, self.c) if self.scheme == FR else None,
            "coeff": decode_coefficients(self.scheme, self.n, self.s, mask),
            "received": self.n - self.s,
            "grad": g,
        }
        self.beta = self.beta - self.lr * g          # beta^(t+1) = beta^(t) - eta g (§III)
        rec["beta"] = self.beta.copy()
        self.t = t + 1
        return rec


# ----------------------------------------------------------------------------
# The paper's baselines on the same problem (§VI-A), literally per worker
# ----------------------------------------------------------------------------

class ISSGDOracle:
    """Ignore-stragglers SGD (§VI-A): every step worker W_i evaluates the
    gradient of its own partition D_i at beta^(t); the master averages the
    gradients of the n - s fastest workers and ignores the rest."""

    def __init__(self, n, s, loss, Xs, ys, lr, beta0=None, K=1):
        self.inner = PGCOracle(CR, n, 0, loss, Xs, ys, lr, beta0=beta0, K=K)   # data, beta, gradients
        self.n, self.s = n, s
        self.t = 0

    @property
    def beta(self):
        return self.inner.beta

    def step(self, mask):
        check_mask(mask, self.n, self.s)
        R = received_set(mask)
        a = np.zeros(self.n)
        for i in R:
            a[i] = 1.0 / len(R)                 # mean of the n - s received gradients
        g = np.zeros_like(self.inner.beta)
        for i in range(self.n):
            gi = self.inner.partition_grad(i)   # stragglers compute too; their result is not used
            if a[i] != 0.0:
                g = g + a[i] * gi
        rec = {"t": self.t, "slot": 0, "eval_partition": list(range(self.n)), "fr_rep": None, "coeff": a,
               "received": len(R), "grad": g}
        self.inner.beta = self.inner.beta - self.inner.lr * g
        rec["beta"] = self.inner.beta.copy()
        self.t += 1
        return rec

    def loss_value(self):
        return self.inner.loss_value()


class GCFROracle:
    """Gradient coding with fractional repetition (§VI-A, the GC baseline; the
    FR construction of §IV-A with every gradient current): every step each
    worker evaluates all c partitions of its group at beta^(t) and uploads
    their sum; the master takes one coded gradient per group, from its
    lowest-index non-straggler, and scales the sum by 1/n."""

    def __init__(self, n, s, loss, Xs, ys, lr, beta0=None, K=1):
        self.inner = PGCOracle(FR, n, 0, loss, Xs, ys, lr, beta0=beta0, K=K)
        self.n, self.s, self.c = n, s, s + 1
        if n % self.c:
            raise ValueError("FR needs c | n")
        self.hold = holdings(FR, n, self.c)
        self.t = 0

    @property
    def beta(self):
        return self.inner.beta

    def step(self, mask):
        check_mask(mask, self.n, self.s)
        coded = [sum(self.inner.partition_grad(k) for k in self.hold[i]) for i in range(self.n)]
        reps = fr_representatives(mask, self.n, self.c)
        a = np.zeros(self.n)
        for r in reps:
            a[r] = 1.0 / self.n
        g = np.zeros_like(self.inner.beta)
        for r in reps:
            g = g + a[r] * coded[r]
        rec = {"t": self.t, "slot": -1, "eval_partition": [-1] * self.n, "fr_rep": reps, "coeff": a,
               "received": self.n - self.s, "grad": g}
        self.inner.beta = self.inner.beta - self.inner.lr * g
        rec["beta"] = self.inner.beta.copy()
        self.t += 1
        return rec

    def loss_value(self):
        return self.inner.loss_value()


class NaiveCROracle(PGCOracle):
    """The naive PGC-CR construction of §V-A (pipelined=True): PGC-CR's
    rotation and stores, GC-CR's weighted uploads and decode weights.  With
    pipelined=False every worker evaluates all c partitions every step: GC
    with cyclic repetition, the exact scheme the naive one pipelines.

    draws: the construction's random numbers, [s][n-1] (reading R15).
    """

    def __init__(self, n, s, loss, Xs, ys, lr, draws=None, beta0=None, K=1, pipelined=True):
        super().__init__(CR, n, s, loss, Xs, ys, lr, beta0=beta0, K=K)
        self.B = gc_cr_encoding(n, s, draws)
        self.C = encoding_coefficients(self.B, self.c)
        self.pipelined = pipelined

    def evaluate(self):
        if self.pipelined or self.t == 0:
            return super().evaluate()
        for i in range(self.n):                       # GC: all c partitions at beta^(t)
            for l in range(self.c):
                self.ring[i][l] = self.partition_grad(self.hold[i][l])
                self.ring_step[i][l] = self.t

    def coded(self, i):
        """W_i's upload: sum_l c_{i,l} * its latest copy of g_{(i+l) mod n} (§V-A)."""
        return sum(self.C[i][l] * self.ring[i][l] for l in range(self.c))

    def decode(self, mask):
        """(1/n) sum_m d_m(J) coded_{j_m} (§V-A; the 1/n is reading R14)."""
        d = gc_decode_weights(self.B, mask)
        g = np.zeros_like(self.beta)
        for i in received_set(mask):
            g = g + (d[i] / self.n) * self.coded(i)
        return g

    def step(self, mask):
        d = gc_decode_weights(self.B, mask)
        alpha = decoding_alpha(self.B, d, mask, self.c)
        rec = super().step(mask)
        if not self.pipelined:
            rec["slot"] = -1
            rec["eval_partition"] = [-1] * self.n
        rec["coeff"] = d / self.n
        rec["d"] = d
        rec["alpha"] = alpha
        rec["alpha_max"] = max(alpha.values())
        rec["alpha_min"] = min(alpha.values())
        return rec


def run_mode(mode, scheme, n, s, loss, Xs, ys, lr, masks, beta0=None, K=1, record_loss=True, draws=None):
    """run() for a training mode: "pgc", "is_sgd", "gc" (GC with FR placement,
    or with CR placement and GC-CR's coefficients when scheme is CR) or
    "naive_cr" (§V-A)."""
    if mode == "pgc":
        return run(scheme, n, s, loss, Xs, ys, lr, masks, beta0=beta0, K=K, record_loss=record_loss)
    if mode == "naive_cr" or (mode == "gc" and scheme == CR):
        o = NaiveCROracle(n, s, loss, Xs, ys, lr, draws=draws, beta0=beta0, K=K, pipelined=mode == "naive_cr")
    else:
        cls = {"is_sgd": ISSGDOracle, "gc": GCFROracle}[mode]
        o = cls(n, s, loss, Xs, ys, lr, beta0=beta0, K=K)
    out = []
    for mask in masks:
        lv = o.loss_value() if record_loss else None
        rec = o.step(mask)
        rec["loss"] = lv
        out.append(rec)
    return out


def run(scheme, n, s, loss, Xs, ys, lr, masks, beta0=None, K=1, record_loss=True):
    """Run len(masks) steps; returns the per-step records with F(beta^(t)) added."""
    o = PGCOracle(scheme, n, s, loss, Xs, ys, lr, beta0=beta0, K=K)
    out = []
    for mask in masks:
        lv = o.loss_value() if record_loss else None
        rec = o.step(mask)
        rec["loss"] = lv
        out.append(rec)
    return out


def all_masks(n: int, s: int):
    """Every straggler mask with exactly s ones (brute force, tiny n)."""
    for S in itertools.combinations(range(n), s):
        m = [0] * n
        for i in S:
            m[i] = 1
        yield m


def binom(n: int, k: int) -> int:
    return math.comb(n, k)
