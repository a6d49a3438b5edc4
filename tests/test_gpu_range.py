"""Cache values beyond the fp16 range. The kernels convert cache keys (and, except in
the bf16 tensor-core attention, values) to fp16; a finite bf16 or fp32 value beyond
+-65504 would become an infinity there and turn the softmax of its rows into NaN.
Such a value is a device-side error instead: the status becomes FSX_ERR_RANGE and the
tick writes no waypoint, like a tick over bad offsets; the next tick over an
in-range cache runs normally and matches the oracle."""
from __future__ import annotations

import numpy as np
import pytest
import torch

from paper_2607_15621_gb300 import fsx, synth

import fsx_cases as fc

pytestmark = pytest.mark.gpu

SMALL = synth.Dims(n_layers=4)
PLANTED = [(3, 5, 7), (10, 5, 70), (20, 17, 1)]  # (row, head, dim) of vehicle 0's layer-2 keys


# B = 1: the single-launch tick; B = 2: the mma.sync split-KV attention; B = 6 (bf16):
# the tensor-core attention
@pytest.mark.parametrize("B,dtype", [(1, "bf16"), (2, "bf16"), (6, "bf16"), (1, "fp32"), (2, "fp32")])
def test_out_of_range_cache_keys_abandon_the_tick(B, dtype):
    lengths = [40 + 13 * b for b in range(B)]
    case = fc.Case(SMALL, lengths, dtype, seed=7)
    clean_k2 = case.k[2].clone()
    for row, head, dim in PLANTED:  # 1e6 is finite in bf16 and fp32, beyond fp16
        case.k[2][row, head, dim] = 1.0e6
    ex = case.expert()
    try:
        out = torch.full((B, SMALL.n_waypoints, 2), 123.0, device="cuda")
        ex.tick(case.k, case.v, case.offsets, case.frames, out)
        torch.cuda.synchronize()
        assert ex.status() == fsx.FSX_ERR_RANGE
        assert torch.all(out == 123.0)  # no waypoint written, no NaN handed out
        # the read cleared the status; the same handle over the in-range cache matches the oracle
        case.k[2].copy_(clean_k2)
        wp = fc.run_tick(ex, case)
    finally:
        ex.close()
    for b in range(B):
        ref, _ = case.oracle_vehicle(b)
        assert np.linalg.norm(wp[b] - ref[0]) <= fc.WAYPOINT_TOL * np.linalg.norm(ref[0]), b


def test_out_of_range_cache_values_are_caught_where_converted():
    """Values are converted to fp16 by the split-KV attention (B = 2 here) and the
    single-launch tick (B = 1)."""
    for lengths in ([30, 50], [50]):
        case = fc.Case(SMALL, lengths, "bf16", seed=8)
        case.v[1][len(lengths) * 17 % sum(lengths), 2, 9] = -3.0e5
        ex = case.expert()
        try:
            out = torch.full((len(lengths), SMALL.n_waypoints, 2), 123.0, device="cuda")
            ex.tick(case.k, case.v, case.offsets, case.frames, out)
            torch.cuda.synchronize()
            assert ex.status() == fsx.FSX_ERR_RANGE
            assert torch.all(out == 123.0)
        finally:
            ex.close()
