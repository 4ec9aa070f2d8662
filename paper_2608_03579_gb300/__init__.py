"""SALT serving hot path on GB300 (sm_103a).

Pinned high-rank domain centroids plus swapped-in ultra-low-rank user
residuals, applied to every token of a heterogeneous batch:

    y += s_c * (x A_c) B_c + s_u * (x a_u) b_u

The compute runs in the CUDA library ``csrc/`` builds (``libsalt.so``); the
``salt`` submodule is its ctypes binding.  Importing this package loads
nothing; ``paper_2608_03579_gb300.salt`` loads the library and raises if it
is missing.
"""
__all__ = ["salt", "workloads"]
