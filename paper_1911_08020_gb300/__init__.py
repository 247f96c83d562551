"""DARB (density-adaptive regular-block pruning, arXiv 1911.08020) on GB300.

The library is the C ABI in ``include/darb.h`` (libdarb.so, hand-written CUDA
for sm_103a); ``paper_1911_08020_gb300.darb`` is its thin Python binding and
``paper_1911_08020_gb300.synth`` draws the seeded synthetic workloads.
"""
__all__ = ["darb", "synth", "build"]
