"""GB300-native MALT / MALTER optimizer step (per-matrix update of every 2-D
weight), implemented as hand-written CUDA for sm_103a behind a C ABI.

The Python side only marshals arguments: see `malt.MaltOptimizer`.
Importing the package does not load the shared library; the first use does,
and fails loudly when it is missing."""
__all__ = ["inputs"]
