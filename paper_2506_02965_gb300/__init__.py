"""GB300-native (sm_103a) sparse MoE expert layer of PC-MoE (arXiv 2506.02965).

The compute lives in the CUDA library ``libmoe.so`` built from ``csrc/``; this
package holds its ctypes binding (``_lib``, same names as include/moe.h) and the
layer driver (``layer.MoELayer``). Importing the binding without the built library
raises: there is no CPU fallback.
"""
import os

LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libmoe.so")


def lib():
    """The ctypes binding (imports libmoe.so; raises ImportError if it is not built)."""
    from . import _lib
    return _lib
