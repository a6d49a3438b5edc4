"""The paper's ten-token expert (Sec. 3.1: state token from the ego state, four visual
tokens, five waypoint queries, two-layer head) through the C ABI against its fp64
oracle on the same seeded inputs: waypoints within 1e-2 relative L2 per vehicle, on
every schedule of the tick (one vehicle: the single-launch tick plus the head launch;
two vehicles: the split-KV attention graph; six: the tensor-core attention graph)."""
from __future__ import annotations

import numpy as np
import pytest
import torch

from oracle import paper_tokens_oracle
from paper_2607_15621_gb300 import fsx, synth

import fsx_cases as fc

pytestmark = pytest.mark.gpu

DIMS = synth.Dims(n_layers=4, n_action=5, n_frame=5)


def _run(lengths, dtype, seed, dims=DIMS):
    B = len(lengths)
    w = synth.make_paper_weights(dims, seed, dtype)
    k, v, off = synth.make_cache(dims, lengths, seed, dtype)
    visual, state = synth.make_paper_inputs(dims, B, seed, dtype)
    ex = fsx.PaperExpert(dims, w, B, max(int(off[-1]), 1), dtype, dtype)
    try:
        out = torch.full((B, 5, 2), float("nan"), device="cuda")
        ex.paper_tick([t.cuda() for t in k], [t.cuda() for t in v], torch.as_tensor(off, device="cuda"),
                      visual.cuda(), state.cuda(), out)
        torch.cuda.synchronize()
        assert ex.status() == fsx.FSX_OK
        launches = ex.launches(B)
        got = out.cpu().double().numpy()
    finally:
        ex.close()
    ref = paper_tokens_oracle.expert_tick_paper_tokens(
        w, [synth.as_f64(t) for t in k], [synth.as_f64(t) for t in v], off, synth.as_f64(visual),
        state.double().numpy(), dims.n_heads, dims.head_dim)
    return got, ref, launches


@pytest.mark.parametrize("lengths,dtype", [([224], "bf16"), ([0], "bf16"), ([96], "fp32"), ([37, 150], "bf16"),
                                           ([20, 0, 64, 130, 5, 90], "bf16")])
def test_paper_tokens_tick_matches_the_oracle(lengths, dtype):
    got, ref, launches = _run(lengths, dtype, seed=3)
    assert np.isfinite(got).all()
    if len(lengths) == 1:
        assert launches == 2  # single-launch tick + two-layer head
    for b in range(len(lengths)):
        err = np.linalg.norm(got[b] - ref[b]) / np.linalg.norm(ref[b])
        assert err <= fc.WAYPOINT_TOL, (b, err)


def test_paper_tokens_full_depth_one_vehicle():
    """All 32 layers at the paper-shaped cache (64 instruction + 40 frames x 4)."""
    dims = synth.Dims(n_action=5, n_frame=5)
    got, ref, _ = _run([224], "bf16", seed=5, dims=dims)
    err = np.linalg.norm(got[0] - ref[0]) / np.linalg.norm(ref[0])
    assert err <= fc.WAYPOINT_TOL, err


def test_the_ego_state_reaches_the_waypoints():
    """Changing only the ego state changes every vehicle's waypoints (the state token is
    attended by the queries at every layer)."""
    dims = DIMS
    w = synth.make_paper_weights(dims, 9, "bf16")
    k, v, off = synth.make_cache(dims, [50, 80], 9, "bf16")
    visual, state = synth.make_paper_inputs(dims, 2, 9, "bf16")
    ex = fsx.PaperExpert(dims, w, 2, int(off[-1]))
    try:
        outs = []
        for s in (state, state + 1.0):
            out = torch.empty(2, 5, 2, device="cuda")
            ex.paper_tick([t.cuda() for t in k], [t.cuda() for t in v], torch.as_tensor(off, device="cuda"),
                          visual.cuda(), s.cuda(), out)
            torch.cuda.synchronize()
            outs.append(out.cpu())
        assert ex.status() == fsx.FSX_OK
    finally:
        ex.close()
    assert (outs[0] - outs[1]).abs().amax(dim=(1, 2)).min() > 1e-3
