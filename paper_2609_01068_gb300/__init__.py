"""OUTLETS length-prediction forward on GB300 (sm_103a).

The compute path lives in the CUDA library built from ``csrc/``; ``outlets``
is its thin ctypes binding.  Importing the package loads nothing; call
``outlets.load()`` (done by the binding on first use).
"""
__all__ = ["outlets", "synth"]
