"""Band-GGNN for GB300: GGNN message propagation on RCM-reordered, block-tridiagonal supergraphs
(arXiv 1906.11786) as hand-written sm_103a CUDA kernels behind a C ABI (include/bandggnn.h).

`paper_1906_11786_gb300.lib` is the ctypes binding of libbandggnn.so; `synth` generates seeded
program-shaped inputs.
"""
from . import _binding as lib  # noqa: F401
from . import synth  # noqa: F401

__all__ = ["lib", "synth"]
