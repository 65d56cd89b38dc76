"""GB300-native (sm_103a) implementation of PACE's condense-and-extract hot path.

The compute lives in ``libpace.so`` (hand-written CUDA kernels behind a C ABI,
declared in ``include/pace.h``).  ``paper_2608_27206_gb300.pace`` is the thin
ctypes binding; ``paper_2608_27206_gb300.synth`` draws seeded inputs.  Importing
the package loads nothing: the library is opened on first use of the binding,
and that fails loudly if it has not been built.
"""
__all__ = ["pace", "synth", "build"]
