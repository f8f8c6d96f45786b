"""fp64 CPU oracle for HeteroFold's prefill-free K/V transfer.

Test infrastructure only: used by ``tests/``, ``__graft_entry__.smoke()`` and
the CPU legs of ``bench.py``; never by the product path.
"""
from .heterofold_oracle import *  # noqa: F401,F403
from .heterofold_oracle import CSR  # noqa: F401
