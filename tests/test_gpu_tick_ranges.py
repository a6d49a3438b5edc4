"""fsx_tick_ranges: the tick with an explicit first cache row per vehicle, so that vehicles'
row ranges may leave gaps (room for the slow system's appends) or overlap (prefixes of one
shared cache, as in the staleness-masked forward over a clip, Sec. 3.2). Checked against
the fp64 oracles with the tick's bars (2e-2 * max|ref| per attention row, 1e-2 relative L2
on the waypoints)."""
from __future__ import annotations

import numpy as np
import pytest
import torch

from oracle import fsx_oracle, staleness_oracle
from paper_2607_15621_gb300 import fsx, synth

import fsx_cases as fc

pytestmark = pytest.mark.gpu

SMALL = synth.Dims(n_layers=4)


def _tick(ex, k, v, off, frames, starts=None, debug=False):
    d = ex.dims
    B = int(frames.shape[0])
    out = torch.empty(B, d.n_waypoints, 2, device="cuda")
    att = None
    if debug:
        att = torch.empty(d.n_layers, B * d.n_tok, d.hd, device="cuda", dtype=torch.float16)
        ex.tick_debug(k, v, off, frames, out, att, starts=starts)
    else:
        ex.tick(k, v, off, frames, out, starts=starts)
    torch.cuda.synchronize()
    assert ex.status() == fsx.FSX_OK
    return out.cpu().numpy().astype(np.float64), att


def _check(wp, att, b, ref_wp, ref_att, T):
    rows = att[:, b * T:(b + 1) * T].to("cpu", torch.float64).numpy()
    assert fc.attn_row_errors(rows, ref_att).max() <= fc.ATTN_ROW_TOL
    assert np.linalg.norm(wp[b] - ref_wp) <= fc.WAYPOINT_TOL * np.linalg.norm(ref_wp)


def test_starts_equal_to_offsets_reproduce_the_tick():
    case = fc.Case(SMALL, [30, 0, 75], "bf16", seed=11)
    ex = case.expert()
    try:
        plain, _ = _tick(ex, case.k, case.v, case.offsets, case.frames)
        ranged, _ = _tick(ex, case.k, case.v, case.offsets, case.frames, starts=case.offsets[:-1].contiguous())
    finally:
        ex.close()
    assert np.array_equal(plain, ranged)  # the graph path (B = 3) is deterministic


@pytest.mark.parametrize("lengths,starts", [([100, 0, 300], [0, 500, 1200]), ([50], [1400])])
def test_gapped_ranges_match_the_oracle(lengths, starts):
    """Vehicles in fixed regions of one cache buffer with free rows between them; one
    vehicle runs as the single-launch tick."""
    rows = 1500
    k, v, _ = synth.make_cache(SMALL, [rows], 12, "bf16")
    k = [t.cuda() for t in k]
    v = [t.cuda() for t in v]
    B = len(lengths)
    frames = synth.make_frames(SMALL, B, 12, "bf16").cuda()
    off = np.concatenate([[0], np.cumsum(lengths)]).astype(np.int64)
    w = fc.weights(SMALL, 12, "bf16")
    ex = fsx.Expert(SMALL, w, B, rows, "bf16", "bf16")
    try:
        wp, att = _tick(ex, k, v, torch.as_tensor(off, device="cuda"), frames,
                        starts=torch.tensor(starts, dtype=torch.int64, device="cuda"), debug=True)
    finally:
        ex.close()
    for b in range(B):
        s, L = starts[b], lengths[b]
        ref_wp, ref_att = fsx_oracle.expert_tick(
            w, [t[s:s + L].float().cpu().numpy() for t in k], [t[s:s + L].float().cpu().numpy() for t in v],
            np.array([0, L]), frames[b:b + 1].double().cpu().numpy(), SMALL.n_heads, SMALL.head_dim,
            SMALL.n_waypoints, capture_attention=True)
        _check(wp, att, b, ref_wp[0], ref_att, SMALL.n_tok)


def test_staleness_clip_forward_matches_the_oracle():
    """All frames of a clip in one tick: block j reads the prefix of the clip's cache that
    ends delta frames earlier (Sec. 3.2); the blocks' ranges overlap."""
    text, tpf, J, delta = 64, 4, 5, 1
    rows = text + tpf * J
    k, v, _ = synth.make_cache(SMALL, [rows], 13, "bf16")
    k = [t.cuda() for t in k]
    v = [t.cuda() for t in v]
    frames = synth.make_frames(SMALL, J, 13, "bf16").cuda()
    prefix = [staleness_oracle.visible_prefix(j, delta, text, tpf) for j in range(J)]
    off = np.concatenate([[0], np.cumsum(prefix)]).astype(np.int64)
    w = fc.weights(SMALL, 13, "bf16")
    ex = fsx.Expert(SMALL, w, J, rows, "bf16", "bf16")
    try:
        wp, att = _tick(ex, k, v, torch.as_tensor(off, device="cuda"), frames,
                        starts=torch.zeros(J, dtype=torch.int64, device="cuda"), debug=True)
    finally:
        ex.close()
    ref_wp, ref_att = staleness_oracle.staleness_masked_forward(
        w, [t.float().cpu().numpy() for t in k], [t.float().cpu().numpy() for t in v], text,
        frames.double().cpu().numpy(), delta, SMALL.n_heads, SMALL.head_dim, SMALL.n_waypoints, tpf,
        capture_attention=True)
    for j in range(J):
        _check(wp, att, j, ref_wp[j], ref_att[j], SMALL.n_tok)


@pytest.mark.parametrize("case", ["past_end", "negative_start", "decreasing_offsets"])
@pytest.mark.parametrize("B", [1, 2])
def test_ranges_outside_the_cache_are_rejected(B, case):
    """A range the cache does not hold sets the status word and the tick writes no
    waypoint (the single-launch and the graph path): a start row whose range runs past
    max_total_cache_tokens, a negative start row, and offsets that decrease (a negative
    length) while start rows are given."""
    rows = 100
    k, v, _ = synth.make_cache(SMALL, [rows], 14, "bf16")
    k = [t.cuda() for t in k]
    v = [t.cuda() for t in v]
    frames = synth.make_frames(SMALL, B, 14, "bf16").cuda()
    w = fc.weights(SMALL, 14, "bf16")
    ex = fsx.Expert(SMALL, w, B, rows, "bf16", "bf16")
    try:
        good_off = [0] + [20 * (i + 1) for i in range(B)]
        if case == "past_end":  # vehicle 0 reads rows 90 .. 109 of a 100-row cache
            off_l, starts_l = good_off, [90] + [0] * (B - 1)
        elif case == "negative_start":
            off_l, starts_l = good_off, [-4] + [0] * (B - 1)
        else:  # the last vehicle's length is -10
            off_l, starts_l = good_off[:-1] + [good_off[-2] - 10], [0] * B
        off = torch.tensor(off_l, dtype=torch.int64, device="cuda")
        starts = torch.tensor(starts_l, dtype=torch.int64, device="cuda")
        out = torch.full((B, SMALL.n_waypoints, 2), 123.0, device="cuda")
        ex.tick(k, v, off, frames, out, starts=starts)
        assert ex.status() == fsx.FSX_ERR_DEVICE_ARG
        assert torch.all(out == 123.0)
        ok = torch.zeros(B, dtype=torch.int64, device="cuda")
        off = torch.tensor(good_off, dtype=torch.int64, device="cuda")
        wp, _ = _tick(ex, k, v, off, frames, starts=ok)
        assert np.isfinite(wp).all()
    finally:
        ex.close()
