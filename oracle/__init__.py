"""fp64 CPU oracle for the BitsMoE quantized MoE-layer forward.

Test infrastructure only: imported by tests/, __graft_entry__.smoke() and the
CPU-baseline / reference legs of bench.py, never by the CUDA library or its
Python binding.
"""
from .bitsmoe_oracle import *  # noqa: F401,F403
from . import bitsmoe_oracle as core  # noqa: F401
from . import quantizer, allocator, calibration  # noqa: F401,E402
from .quantizer import quantize_units  # noqa: F401,E402
