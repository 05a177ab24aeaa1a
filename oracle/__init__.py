"""fp64 CPU oracle of Pipelined Gradient Coding; test infrastructure only.

Only the tests, ``__graft_entry__.smoke()`` and the CPU legs of ``bench.py``
may import this package.  The product path never does.
"""

from .pgc_oracle import *  # noqa: F401,F403
