"""fp64 CPU oracle for the role-conditional KV-eviction hot path.

Test infrastructure only: imported by ``tests/``, ``__graft_entry__.smoke()``
and the CPU-baseline leg of ``bench.py``.  The library (``librolekv.so`` and
its Python binding) never imports, links or runs anything in this package.
"""
from . import rolekv_oracle  # noqa: F401
