"""CPU oracle for the XShare MoE-layer forward.

TEST INFRASTRUCTURE ONLY: imported by the tests, by ``__graft_entry__.smoke()``
and by the CPU-baseline leg of ``bench.py``; never by the product package.
"""
from . import xshare_oracle  # noqa: F401
