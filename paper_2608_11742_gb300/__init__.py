"""GB300-native scoring path of Ripple-Pivot Search (RPS).

The CUDA library (``librps.so``) and its ctypes binding live in ``rps``; importing
that module loads the library and raises if it is missing. ``synth`` and
``configs`` are pure numpy and import without a GPU.
"""
__all__ = ["rps", "synth", "configs"]
