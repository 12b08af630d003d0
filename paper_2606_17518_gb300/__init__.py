"""GB300 (sm_103a) fork-decode attention over a shared reasoning prefix.

The compute lives in ``libspecgen.so`` (CUDA kernels behind the C ABI of
``include/specgen.h``); ``_lib`` is its ctypes binding and ``fork_attn`` a
torch-buffer convenience wrapper.  ``workloads`` builds seeded synthetic
inputs.  Importing the package has no side effects.
"""

__all__ = ["build", "workloads", "fork_attn", "_lib"]
