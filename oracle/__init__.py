"""Independent CPU oracle of the LR-QAT linear layer (test infrastructure only).

Only the tests, ``__graft_entry__.smoke`` and the CPU-baseline leg of
``bench.py`` use this package; the library never imports it.
"""
from .lrqat_oracle import *  # noqa: F401,F403
from .lrqat_oracle import Layer, PHI_QFIXED, PHI_INT_PACKED, FLOAT_PHI  # noqa: F401
