"""NOBLE linear layer (arXiv 2603.06492) with the CosNet branch on GB300.

The compute path is the C-ABI library ``libnoble.so`` built from ``csrc/``
(hand-written sm_103a kernels); ``binding`` is a thin ctypes layer over it.
Importing this package does not load the library; ``binding.load()`` does and
raises if it is missing.
"""
__all__ = ["binding", "inputs", "build"]
