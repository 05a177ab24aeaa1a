"""GB300-native hot path of Pipelined Gradient Coding (PGC).

The compute lives in ``libpgc.so`` (CUDA for sm_103a behind a C ABI declared
in ``include/pgc.h``).  ``paper_2607_20739_gb300.binding`` is the thin ctypes
layer over it; ``paper_2607_20739_gb300.workloads`` draws seeded inputs.

The binding is imported lazily so that the input generators can be used on a
machine where the library has not been built; any use of the binding without
the library raises immediately.
"""

__all__ = ["binding", "workloads", "PGC", "PGCError"]


def __getattr__(name):
    if name in ("PGC", "PGCError"):
        from . import binding
        return getattr(binding, name)
    if name in ("binding", "workloads"):
        import importlib
        return importlib.import_module(f".{name}", __name__)
    raise AttributeError(name)
