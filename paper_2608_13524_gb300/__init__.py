"""GB300 (sm_103a) DARTree draft-tree construction.

The hot path is hand-written CUDA behind the C ABI in include/dart.h; the
Python module ``dart`` is a thin ctypes binding of it.
"""
from . import dart  # noqa: F401
from .dart import Dart  # noqa: F401
