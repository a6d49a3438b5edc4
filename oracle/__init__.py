"""fp64 CPU oracles (test infrastructure only).

fsx_oracle     the action-expert tick (Sec. 3.1, Eq. 1);
append_oracle  the backbone's incremental four-token cache append and the
               monolithic forward it must match (Sec. 1, Sec. 3.3);
paper_tokens_oracle  the tick with the paper's own ten-token layout (state
               MLP, four visual tokens, five queries, two-layer head);
staleness_oracle  the staleness-masked forward over a training clip (Sec. 3.2).

Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline / reference
legs may import this package; the product path never does.
"""
from .fsx_oracle import (RMS_EPS, attention_eq1, expert_tick, rms_norm, silu,
                         softmax_row_sums)

__all__ = ["RMS_EPS", "attention_eq1", "expert_tick", "rms_norm", "silu",
           "softmax_row_sums"]
