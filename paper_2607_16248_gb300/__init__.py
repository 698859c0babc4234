"""GB300-native low-bit KV-cache decode step with DGAP local distribution
restoration (arXiv 2607.16248).

The compute path is ``libkvq.so`` (CUDA, sm_103a) behind the C ABI of
``include/kvq.h``; ``kvq`` is its thin Python binding and ``synth`` the seeded
synthetic inputs.  Importing this package loads nothing; the library is
loaded on first use.
"""

__all__ = ["kvq", "synth", "build"]
