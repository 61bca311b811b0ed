"""fp64 CPU oracle of the rollout / re-scoring hot path.

Test infrastructure only: imported by tests/, __graft_entry__.smoke() and the CPU
baseline leg of bench.py, never by the product library or its Python binding.
"""
from .vla_oracle import *  # noqa: F401,F403
from .vla_oracle import Oracle, Shape, Weights, action_head, bin_centre, full_forward, shape_from  # noqa: F401
