"""GB300-native grouped ternary (W1.58A16) linear layer.

``tq`` is the ctypes binding of libtq (include/tq.h); ``synth`` draws the seeded
synthetic inputs; ``build`` compiles libtq.so for sm_103a.
"""
from . import synth  # noqa: F401

__all__ = ["synth", "tq", "build"]


def __getattr__(name):
    if name in ("tq", "build"):
        import importlib
        return importlib.import_module(f".{name}", __name__)
    raise AttributeError(name)
