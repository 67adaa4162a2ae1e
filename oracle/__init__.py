"""Float64 CPU oracle of the expert-choice MoE layer (test infrastructure only).

Only tests/, __graft_entry__.smoke() and bench.py's CPU baseline leg use it.
"""
from . import ecmoe  # noqa: F401
