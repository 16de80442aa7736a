"""GB300-native evaluation of CNNs under dynamic fixed-point configurations (FxP-QNet hot path).

libfxpq.so (hand-written sm_103a CUDA behind the C ABI in include/fxpq.h) does every step; this
package is its Python binding (``fxpq``) and the host-side network planner (``net``).
"""
from . import build  # noqa: F401
