"""Block-sparse pruned-layer inference on GB300 (sm_103a).

The compute path is the C-ABI library ``libbp.so`` (hand-written CUDA, built
from ``csrc/``); ``paper_2111_11581_gb300.bp`` is its thin ctypes binding.
Importing this package loads nothing: the library is opened on first use and
an error is raised if it is missing.  There is no CPU fallback.
"""
__all__ = ["bp", "inputs"]
