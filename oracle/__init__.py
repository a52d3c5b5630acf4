"""fp64 CPU oracle of the MLA decode step -- test infrastructure only.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline / reference
arm of ``bench.py`` may import this package.  It shares no code with the CUDA
library in ``paper_2607_27269_gb300``.
"""
