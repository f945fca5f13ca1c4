"""GB300-native (sm_103a) engine for ZeroLock's decoupled per-chunk update.

The compute path is libzerolock.so (hand-written CUDA behind the C ABI of
include/zerolock.h); ``binding`` is its ctypes binding. Build with
``paper_2608_07974_gb300._build.build()``.
"""
from ._build import build  # noqa: F401


def load():
    """Import the binding (raises ImportError if the library is not built)."""
    from . import binding
    return binding
