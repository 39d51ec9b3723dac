"""GB300-native fused decode of binary-spherical-coded LLM weights (BiSCo-LLM).

The compute path is the C-ABI CUDA library ``libbisco.so`` built from
``csrc/``; :mod:`.bisco` is its thin ctypes binding and :mod:`.synth` draws
seeded synthetic inputs.  Importing the package loads nothing.
"""
__all__ = ["bisco", "synth", "build"]
