"""GB300-native grouped ternary (W1.58A16) linear layer.

``tq`` is the ctypes binding of libtq (include/tq.h); ``ternary_linear`` wraps it as a
torch autograd function and module (TernaryLinear, §3.1) and its packed inference
form (PackedTernaryLinear); ``synth`` draws the seeded
synthetic inputs; ``build`` compiles libtq.so for sm_103a.
"""
from . import synth  # noqa: F401

__all__ = ["synth", "tq", "build", "ternary_linear"]


def __getattr__(name):
    if name in ("tq", "build", "ternary_linear"):
        import importlib
        return importlib.import_module(f".{name}", __name__)
    raise AttributeError(name)
