"""GB300-native decode step of T-LoopFormer (token-level elastic-depth looped transformer).

The compute path is the CUDA library ``libtlf.so`` built from ``csrc/`` for
sm_103a; ``tlf`` is its ctypes binding and ``synth`` the seeded input
generator. Importing the package loads nothing: the library is loaded on the
first use of ``tlf``.
"""
__all__ = ["synth", "tlf"]
