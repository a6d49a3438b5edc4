"""fp64 CPU oracle of the action-expert tick (test infrastructure only).

Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline / reference
legs may import this package; the product path never does.
"""
from .fsx_oracle import (RMS_EPS, attention_eq1, expert_tick, rms_norm, silu,
                         softmax_row_sums)

__all__ = ["RMS_EPS", "attention_eq1", "expert_tick", "rms_norm", "silu",
           "softmax_row_sums"]
