"""ORACLE -- test infrastructure, not part of the product.

A plain, slow CPU restatement of Gradient Energy Matching (arXiv 1805.08469) written in
C++ (``*.cpp`` in this folder) and loaded through ctypes.  Only the tests, the smoke
check and the CPU-baseline leg of the benchmark import it.  It shares no code with the
CUDA path, and the CUDA path never imports it.
"""
from .oracle import *  # noqa: F401,F403
