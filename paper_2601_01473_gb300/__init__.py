"""GB300-native AGNES data-preparation path (arXiv 2601.01473): block-wise,
hyperbatch-based multi-hop neighbour sampling and feature gathering in CUDA
kernels for sm_103a behind a C ABI (include/agnes.h).  ``agnes`` is the thin
ctypes binding; ``build`` compiles the library in place."""
from .agnes import AgnesError, Graph, Hop, MinibatchView, lib

__all__ = ["AgnesError", "Graph", "Hop", "MinibatchView", "lib"]
