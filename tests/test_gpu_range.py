"""Cache values beyond the fp16 range. The kernels convert cache keys (and, except in
the bf16 tensor-core attention, values) to fp16; a finite bf16 or fp32 value beyond
+-65504 would become an infinity there and turn the softmax of its rows into NaN.
Every conversion saturates instead and raises FSX_ERR_RANGE, so a tick over such a
cache completes, equals the oracle on the saturated cache, and reports the fact."""
from __future__ import annotations

import numpy as np
import pytest
import torch

from oracle import fsx_oracle
from paper_2607_15621_gb300 import fsx, synth

import fsx_cases as fc

pytestmark = pytest.mark.gpu

SMALL = synth.Dims(n_layers=4)
F16_MAX = 65504.0
PLANTED = [(3, 5, 7), (10, 5, 70), (20, 17, 1)]  # (row, head, dim) of vehicle 0's layer-2 keys


def _oracle_saturated(case, b, layer):
    lo, hi = int(case.offsets_np[b]), int(case.offsets_np[b + 1])
    k = [t[lo:hi].to("cpu", torch.float32).numpy().copy() for t in case.k]
    v = [t[lo:hi].to("cpu", torch.float32).numpy() for t in case.v]
    k[layer] = np.clip(k[layer], -F16_MAX, F16_MAX)
    fr = case.frames[b:b + 1].to("cpu", torch.float64).numpy()
    d = case.dims
    wp, _ = fsx_oracle.expert_tick(case.w, k, v, np.array([0, hi - lo]), fr, d.n_heads, d.head_dim, d.n_waypoints,
                                   capture_attention=True)
    return wp[0]


# B = 1: the single-launch tick; B = 2: the mma.sync split-KV attention; B = 6 (bf16):
# the tensor-core attention
@pytest.mark.parametrize("B,dtype", [(1, "bf16"), (2, "bf16"), (6, "bf16"), (1, "fp32"), (2, "fp32")])
def test_out_of_range_cache_keys_are_saturated_and_flagged(B, dtype):
    lengths = [40 + 13 * b for b in range(B)]
    case = fc.Case(SMALL, lengths, dtype, seed=7)
    for row, head, dim in PLANTED:  # 1e6 is finite in bf16 and fp32, beyond fp16
        case.k[2][row, head, dim] = 1.0e6
    ex = case.expert()
    try:
        out = torch.full((B, SMALL.n_waypoints, 2), float("nan"), device="cuda")
        ex.tick(case.k, case.v, case.offsets, case.frames, out)
        torch.cuda.synchronize()
        assert ex.status() == fsx.FSX_ERR_RANGE
        wp = out.cpu().numpy().astype(np.float64)
        assert np.isfinite(wp).all()
        ref = _oracle_saturated(case, 0, 2)
        assert np.linalg.norm(wp[0] - ref) <= fc.WAYPOINT_TOL * np.linalg.norm(ref)
        # the read cleared the flag; the same handle over an in-range cache reports OK
        clean = fc.Case(SMALL, lengths, dtype, seed=7)
        out2 = torch.empty_like(out)
        ex.tick(clean.k, clean.v, clean.offsets, clean.frames, out2)
        torch.cuda.synchronize()
        assert ex.status() == fsx.FSX_OK
        assert torch.isfinite(out2).all()
    finally:
        ex.close()


def test_out_of_range_cache_values_are_flagged_where_converted():
    """Values are converted to fp16 by the split-KV attention (B = 2 here)."""
    case = fc.Case(SMALL, [30, 50], "bf16", seed=8)
    case.v[1][35, 2, 9] = -3.0e5
    ex = case.expert()
    try:
        out = torch.empty(2, SMALL.n_waypoints, 2, device="cuda")
        ex.tick(case.k, case.v, case.offsets, case.frames, out)
        torch.cuda.synchronize()
        assert ex.status() == fsx.FSX_ERR_RANGE
        assert torch.isfinite(out).all()
    finally:
        ex.close()
