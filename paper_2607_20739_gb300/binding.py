"""Thin ctypes binding of libpgc (include/pgc.h): argument marshalling only.

Every step of the hot path runs in the library's CUDA kernels.  Importing
this module loads ``_lib/libpgc.so`` and raises ``ImportError`` if it is
missing: there is no CPU fallback.

Arrays may be numpy arrays (host memory) or torch tensors (device memory,
passed by pointer).  Streams are torch streams or raw ``cudaStream_t``
integers.
"""

from __future__ import annotations

import ctypes as C
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_lib", "libpgc.so")

if not os.path.exists(LIB_PATH):
    raise ImportError(f"libpgc.so not built ({LIB_PATH}); run __graft_entry__.build() first")

lib = C.CDLL(LIB_PATH)

OK, EINVAL, EMASK, ESTATE, ENOMEM, ECUDA, ENOTSUP, ETIMEOUT, ESCRATCH, ESINGULAR = 0, -1, -2, -3, -4, -5, -6, -7, -8, -9
FR, CR = 0, 1
LOGISTIC, LSQ, SOFTMAX = 0, 1, 2
F32, BF16 = 0, 1

SCHEMES = {"FR": FR, "CR": CR}
LOSSES = {"logistic": LOGISTIC, "lsq": LSQ, "softmax": SOFTMAX}
DTYPES = {"f32": F32, "bf16": BF16}
MODE_PGC, MODE_IS_SGD, MODE_GC, MODE_NAIVE_CR = 0, 1, 2, 3
MODES = {"pgc": MODE_PGC, "is_sgd": MODE_IS_SGD, "gc": MODE_GC, "naive_cr": MODE_NAIVE_CR}


class StepInfo(C.Structure):
    _fields_ = [("t", C.c_int64), ("slot", C.c_int32), ("received", C.c_int32),
                ("eval_partition", C.POINTER(C.c_int32)), ("fr_rep", C.POINTER(C.c_int32))]


_vp = C.c_void_p
_i32 = C.c_int32
_i64 = C.c_int64
_sig = {
    "pgc_create": (C.c_int, [C.POINTER(_vp), _i32, _i32, _i32, _i32, _i32, _i64, _i64, C.POINTER(_i64), C.c_float,
                             C.POINTER(C.c_float), _vp]),
    "pgc_create_mode": (C.c_int, [C.POINTER(_vp), _i32, _i32, _i32, _i32, _i32, _i32, _i64, _i64, C.POINTER(_i64), C.c_float,
                             C.POINTER(C.c_float), _vp]),
    "pgc_load_partitions": (C.c_int, [_vp, C.POINTER(_vp), C.POINTER(_vp), _i32]),
    "pgc_step": (C.c_int, [_vp, _vp, _vp, _vp, _i32, C.POINTER(StepInfo)]),
    "pgc_loss": (C.c_int, [_vp, C.POINTER(C.c_double)]),
    "pgc_sync": (C.c_int, [_vp]),
    "pgc_destroy": (C.c_int, [_vp]),
    "pgc_strerror": (C.c_char_p, [_i32]),
    "pgc_last_cuda_error": (C.c_char_p, []),
    "pgc_gradient_path": (C.c_char_p, [_vp]),
    "pgc_placement": (C.c_int, [_i32, _i32, _i32, C.POINTER(_i32)]),
    "pgc_schedule": (C.c_int, [_i32, _i32, _i32, _i64, C.POINTER(_i32), C.POINTER(_i32)]),
    "pgc_get_store": (C.c_int, [_vp, _i32, _i32, C.POINTER(C.c_float)]),
    "pgc_checkpoint_bytes": (C.c_int, [_vp, C.POINTER(_i64)]),
    "pgc_checkpoint_save": (C.c_int, [_vp, _vp, _i64]),
    "pgc_checkpoint_load": (C.c_int, [_vp, _vp, _i64]),
    "pgc_get_store_cols": (C.c_int, [_vp, _i32, _i32, _i64, _i64, C.POINTER(C.c_float)]),
    "pgc_get_decode": (C.c_int, [_vp, C.POINTER(C.c_float)]),
    "pgc_set_gc_encoding": (C.c_int, [_vp, C.POINTER(C.c_double)]),
    "pgc_get_gc_encoding": (C.c_int, [_vp, C.POINTER(C.c_double)]),
    "pgc_get_gc_decode": (C.c_int, [_vp, C.POINTER(C.c_double), C.POINTER(C.c_double)]),
    "pgc_get_weights": (C.c_int, [_vp, C.POINTER(C.c_float)]),
    "pgc_set_weights": (C.c_int, [_vp, C.POINTER(C.c_float)]),
    "pgc_step_count": (C.c_int64, [_vp]),
    "pgc_timing": (C.c_int, [_vp, _i32]),
    "pgc_timing_read": (C.c_int, [_vp, C.POINTER(C.c_double), C.POINTER(_i64), C.POINTER(_i64)]),
    "pgc_gradient_noalloc": (C.c_int, [_i32, _i32, _i64, _i64, _vp, _vp, _vp, _vp, _vp]),
}
for _name, (_res, _args) in _sig.items():
    _f = getattr(lib, _name)
    _f.restype = _res
    _f.argtypes = _args

EXPORTED = tuple(_sig)


# kernel groups of one step, in launch order (PGC_KGRAD .. PGC_KDECODE)
KERNEL_GROUPS = ("gradient", "residual", "gradient_backward", "commit", "decode")


class PGCError(RuntimeError):
    def __init__(self, code: int, where: str):
        self.code = code
        msg = f"{where}: {lib.pgc_strerror(code).decode()} ({code})"
        if code in (ECUDA, ENOMEM):
            name = lib.pgc_last_cuda_error().decode()
            if name:
                msg += f" [{name}]"
        super().__init__(msg)


def _check(code: int, where: str) -> None:
    if code != OK:
        raise PGCError(code, where)


def _enum(v, table):
    return table[v] if isinstance(v, str) else int(v)


def _is_torch(x) -> bool:
    return type(x).__module__.startswith("torch")


def _ptr(x):
    """Address of a contiguous numpy array or torch tensor."""
    if _is_torch(x):
        if not x.is_contiguous():
            raise ValueError("tensor must be contiguous")
        return C.c_void_p(x.data_ptr())
    if not x.flags["C_CONTIGUOUS"]:
        raise ValueError("array must be C-contiguous")
    return C.c_void_p(x.ctypes.data)


def _stream_handle(stream) -> int:
    if stream is None:
        return 0
    if hasattr(stream, "cuda_stream"):
        return int(stream.cuda_stream)
    return int(stream)


def placement(scheme, n: int, s: int) -> np.ndarray:
    out = np.zeros(n * (s + 1), dtype=np.int32)
    _check(lib.pgc_placement(_enum(scheme, SCHEMES), n, s, out.ctypes.data_as(C.POINTER(_i32))), "pgc_placement")
    return out.reshape(n, s + 1)


def schedule(scheme, n: int, s: int, t: int):
    out = np.zeros(n, dtype=np.int32)
    slot = _i32(0)
    _check(lib.pgc_schedule(_enum(scheme, SCHEMES), n, s, t, out.ctypes.data_as(C.POINTER(_i32)), C.byref(slot)),
           "pgc_schedule")
    return out, slot.value


class PGC:
    """One PGC run on the current CUDA device (a ``pgc_ctx``)."""

    def __init__(self, scheme, n: int, s: int, loss, dtype, d: int, K: int = 1, rows=None, lr: float = 0.1,
                 w0=None, stream=None, mode="pgc"):
        self.scheme = _enum(scheme, SCHEMES)
        self.loss_kind = _enum(loss, LOSSES)
        self.dtype = _enum(dtype, DTYPES)
        self.mode = _enum(mode, MODES)
        c = 1 if self.mode == MODE_IS_SGD else s + 1
        self.n, self.s, self.c, self.d, self.K = n, s, c, d, K
        rows = np.asarray(rows if rows is not None else [1] * n, dtype=np.int64)
        if rows.shape != (n,):
            raise ValueError("rows must have one entry per partition")
        self.rows = rows
        w0p = None
        if w0 is not None:
            w0 = np.ascontiguousarray(np.asarray(w0, dtype=np.float32).reshape(-1))
            w0p = w0.ctypes.data_as(C.POINTER(C.c_float))
        self._stream = _stream_handle(stream)
        h = _vp()
        _check(lib.pgc_create_mode(C.byref(h), self.mode, n, s, self.scheme, self.loss_kind, self.dtype, d, K,
                                   rows.ctypes.data_as(C.POINTER(_i64)), C.c_float(lr), w0p, _vp(self._stream)),
               "pgc_create_mode")
        self._h = h
        self._mask = np.zeros(n, dtype=np.uint8)
        self._eval = np.zeros(n, dtype=np.int32)
        self._rep = np.zeros(max(1, n // self.c), dtype=np.int32)

    # -- lifetime --------------------------------------------------------
    def close(self):
        if getattr(self, "_h", None) is not None and self._h.value:
            lib.pgc_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    # -- calls -----------------------------------------------------------
    def load(self, Xs, ys, on_device: bool | None = None):
        """Copy partitions (numpy host arrays or torch device tensors)."""
        if len(Xs) != self.n or len(ys) != self.n:
            raise ValueError("need n feature and label arrays")
        if on_device is None:
            on_device = _is_torch(Xs[0]) and Xs[0].is_cuda
        keep = []
        xp = (_vp * self.n)()
        yp = (_vp * self.n)()
        for k in range(self.n):
            X, y = Xs[k], ys[k]
            if not _is_torch(X):
                X = np.ascontiguousarray(X)
                y = np.ascontiguousarray(y)
            keep += [X, y]
            xp[k] = _ptr(X).value
            yp[k] = _ptr(y).value
        _check(lib.pgc_load_partitions(self._h, xp, yp, 1 if on_device else 0), "pgc_load_partitions")

    def step(self, mask, grad_out=None, w_out=None, info: bool = True):
        """One training step.  Outputs may be numpy (host, waits) or torch CUDA
        tensors (device, returns immediately)."""
        m = mask
        if not (type(m) is np.ndarray and m.dtype == np.uint8 and m.flags.c_contiguous):
            m = np.ascontiguousarray(np.asarray(mask, dtype=np.uint8))
        if m.shape != (self.n,):
            raise ValueError("mask must have n entries")
        on_dev = 0
        for o in (grad_out, w_out):
            if o is not None and _is_torch(o) and o.is_cuda:
                on_dev = 1
        gi = None
        if info:
            gi = StepInfo()
            gi.eval_partition = self._eval.ctypes.data_as(C.POINTER(_i32))
            gi.fr_rep = self._rep.ctypes.data_as(C.POINTER(_i32))
        _check(lib.pgc_step(self._h, m.ctypes.data,
                            _ptr(grad_out) if grad_out is not None else None,
                            _ptr(w_out) if w_out is not None else None, on_dev,
                            C.byref(gi) if gi is not None else None), "pgc_step")
        if not info:
            return None
        return {
            "t": gi.t, "slot": gi.slot, "received": gi.received,
            "eval_partition": self._eval.copy(),
            "fr_rep": self._rep.copy() if self.scheme == FR else None,
        }

    @property
    def gradient_path(self) -> str:
        """Name of the kernel path chosen for the per-partition gradients."""
        return lib.pgc_gradient_path(self._h).decode()

    def sync(self):
        _check(lib.pgc_sync(self._h), "pgc_sync")

    def loss(self) -> float:
        v = C.c_double()
        _check(lib.pgc_loss(self._h, C.byref(v)), "pgc_loss")
        return v.value

    def store(self, worker: int, slot: int) -> np.ndarray:
        out = np.zeros(self.K * self.d, dtype=np.float32)
        _check(lib.pgc_get_store(self._h, worker, slot, out.ctypes.data_as(C.POINTER(C.c_float))), "pgc_get_store")
        return out.reshape(self.K, self.d) if self.K > 1 else out

    def decode_coefficients(self) -> np.ndarray:
        out = np.zeros(self.n, dtype=np.float32)
        _check(lib.pgc_get_decode(self._h, out.ctypes.data_as(C.POINTER(C.c_float))), "pgc_get_decode")
        return out

    def set_gc_encoding(self, draws=None) -> None:
        """GC-CR's encoding from the construction's draws [s][n-1] (§V-A)."""
        p = None
        if self.s > 0:
            draws = np.ascontiguousarray(np.asarray(draws, dtype=np.float64).reshape(self.s, self.n - 1))
            p = draws.ctypes.data_as(C.POINTER(C.c_double))
        _check(lib.pgc_set_gc_encoding(self._h, p), "pgc_set_gc_encoding")

    def gc_encoding(self) -> np.ndarray:
        """Encoding coefficients c_{j,l}, shape [n][c]."""
        out = np.zeros((self.n, self.c), dtype=np.float64)
        _check(lib.pgc_get_gc_encoding(self._h, out.ctypes.data_as(C.POINTER(C.c_double))), "pgc_get_gc_encoding")
        return out

    def gc_decode(self):
        """The last step's decode weights d_j(J) [n] and (max, min) of alpha_{m,k}."""
        d = np.zeros(self.n, dtype=np.float64)
        ar = np.zeros(2, dtype=np.float64)
        _check(lib.pgc_get_gc_decode(self._h, d.ctypes.data_as(C.POINTER(C.c_double)),
                                     ar.ctypes.data_as(C.POINTER(C.c_double))), "pgc_get_gc_decode")
        return d, (float(ar[0]), float(ar[1]))

    def store_cols(self, worker: int, slot: int, col0: int, ncols: int) -> np.ndarray:
        """Columns [col0, col0 + ncols) of the flattened K*d stored gradient."""
        out = np.empty(ncols, dtype=np.float32)
        _check(lib.pgc_get_store_cols(self._h, worker, slot, col0, ncols, out.ctypes.data_as(C.POINTER(C.c_float))),
               "pgc_get_store_cols")
        return out

    def checkpoint(self) -> np.ndarray:
        """The run's state (t, beta, stores, slot totals) as a host byte array."""
        nb = _i64()
        _check(lib.pgc_checkpoint_bytes(self._h, C.byref(nb)), "pgc_checkpoint_bytes")
        buf = np.empty(nb.value, dtype=np.uint8)
        _check(lib.pgc_checkpoint_save(self._h, buf.ctypes.data, nb.value), "pgc_checkpoint_save")
        return buf

    def restore(self, buf) -> None:
        """Resume from checkpoint(): the next step is the saved run's next step."""
        b = np.ascontiguousarray(np.asarray(buf, dtype=np.uint8))
        _check(lib.pgc_checkpoint_load(self._h, b.ctypes.data, b.size), "pgc_checkpoint_load")

    def weights(self) -> np.ndarray:
        out = np.zeros(self.K * self.d, dtype=np.float32)
        _check(lib.pgc_get_weights(self._h, out.ctypes.data_as(C.POINTER(C.c_float))), "pgc_get_weights")
        return out.reshape(self.K, self.d) if self.K > 1 else out

    def set_weights(self, w):
        w = np.ascontiguousarray(np.asarray(w, dtype=np.float32).reshape(-1))
        _check(lib.pgc_set_weights(self._h, w.ctypes.data_as(C.POINTER(C.c_float))), "pgc_set_weights")

    def timing(self, enable: bool):
        _check(lib.pgc_timing(self._h, 1 if enable else 0), "pgc_timing")

    def timing_read(self):
        """Per kernel group (KERNEL_GROUPS order): summed ms and launches."""
        ms = (C.c_double * len(KERNEL_GROUPS))()
        nl = (_i64 * len(KERNEL_GROUPS))()
        steps = _i64()
        _check(lib.pgc_timing_read(self._h, ms, nl, C.byref(steps)), "pgc_timing_read")
        return {"ms": list(ms), "launches": list(nl), "steps": steps.value}

    @property
    def t(self) -> int:
        return int(lib.pgc_step_count(self._h))
