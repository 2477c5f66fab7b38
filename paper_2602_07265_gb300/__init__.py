"""XShare MoE-layer forward on GB300 (sm_103a).

The compute lives in ``libxshare.so`` (C ABI, hand-written CUDA kernels); the
``xshare`` module is its thin ctypes binding.  Importing this package does not
load the library; ``paper_2602_07265_gb300.xshare`` does, and raises if the
library has not been built.
"""

__all__ = ["xshare", "workloads"]
