"""GRID's cold full-vocabulary next-token mask on GB300 (sm_103a).

The compute path is ``csrc/`` (host compiler in C++, kernels in CUDA) behind the
C ABI of ``include/grid.h``; ``grid.py`` is its thin ctypes binding and
``build.py`` compiles the shared library in-tree.
"""
from .build import build, library_path  # noqa: F401
