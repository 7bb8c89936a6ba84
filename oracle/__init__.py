"""fp64 CPU oracle of the eviction path.

Test infrastructure: only ``tests/``, ``__graft_entry__.smoke()`` and
``bench.py``'s CPU-baseline leg may import this package.
"""
from .epikv_oracle import *  # noqa: F401,F403
