"""GB300-native (sm_103a) random-Fourier-feature linear attention with learnable
spectral frequencies (Flexformer, stationary and nonstationary variants).

The compute path is the CUDA library ``libflexattn.so`` built from ``csrc/`` behind the
C ABI declared in ``include/flexattn.h``; ``flexattn`` is its thin ctypes binding.
Importing this package loads nothing: the library is opened on first use, and a missing
library is an error, never a fallback.
"""
__all__ = ["flexattn", "workloads"]
