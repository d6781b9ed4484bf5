"""GB300-native beam-decode hot path of thought-level beam search (Gambit).

* ``binding``  - ctypes functions with the C ABI's names (``include/gambit.h``).
* ``pool``     - ``BeamPool``: device buffers from PyTorch, all work in the library.
* ``build``    - nvcc build of ``libgambit.so`` for sm_103a.
"""
from paper_2608_08020_gb300 import binding  # noqa: F401

__all__ = ["binding"]
