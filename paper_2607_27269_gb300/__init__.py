"""GB300-native absorbed multi-head latent attention (MLA) decode step.

The compute lives in ``libgbmla.so`` (hand-written sm_103a CUDA kernels behind a
C ABI, declared in ``include/gbmla.h``).  ``paper_2607_27269_gb300.abi`` is the
thin ctypes binding with the same entry-point names.  Nothing is loaded at
import time, so ``workloads`` can be imported without a GPU.
"""
__all__ = ["abi", "workloads", "build"]
