"""GB300-native world-model dream engine (RLFlow, SIGMOD'22): C ABI + thin binding.

The CUDA library ``libwm.so`` holds every kernel; ``wm`` marshals arguments.
Build it with ``__graft_entry__.build()`` (or ``python -m paper_2205_01435_gb300._build``).
"""
from . import _build  # noqa: F401


def load():
    """Imports the ctypes binding; raises ImportError if libwm.so has not been built."""
    from . import wm
    return wm
