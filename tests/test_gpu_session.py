"""The asynchronous fast-slow schedule (Sec. 3.3, Fig. 1) through the C ABI: one
vehicle's ticks over the committed rows of its cache while appends write the rows
behind them, in the serial and the concurrent schedule. Every tick's waypoints must
equal the tick oracle on exactly the rows of its snapshot (1e-2 relative L2): a tick
that read a row of an append still in flight, or missed a committed one, would
differ. The appended rows must equal the append oracle's (2e-2 of each row's largest
entry), and rows outside the appended ones stay bitwise unchanged."""
from __future__ import annotations

import numpy as np
import pytest
import torch

from oracle import append_oracle, fsx_oracle
from paper_2607_15621_gb300 import fsx, synth

import fsx_cases as fc

pytestmark = pytest.mark.gpu

EXPERT = synth.Dims(n_layers=2)
BACKBONE = synth.BackboneDims(n_layers=2)
L0, CAP = 50, 96


def _setup(concurrent, seed=11):
    k0, v0, _ = synth.make_cache(EXPERT, [L0], seed, "bf16")
    kc = [torch.zeros(CAP, EXPERT.n_heads, EXPERT.head_dim, dtype=torch.bfloat16, device="cuda") for _ in k0]
    vc = [torch.zeros_like(t) for t in kc]
    for dst, src in zip(kc + vc, k0 + v0):
        dst[:L0] = src.cuda()
    w = fc.weights(EXPERT, seed, "bf16")
    bw = synth.make_backbone_weights(BACKBONE, seed, "bf16")
    ex = fsx.Expert(EXPERT, w, 1, CAP)
    ap = fsx.Append(BACKBONE, bw, 1, CAP)
    ses = fsx.Session(ex, ap, kc, vc, CAP, L0, concurrent)
    frames = synth.make_frames(EXPERT, 1, seed, "bf16").cuda()
    return w, bw, kc, vc, ex, ap, ses, frames


def _oracle_tick(w, kc, vc, rows, frames):
    k = [t[:rows].float().cpu().numpy() for t in kc]
    v = [t[:rows].float().cpu().numpy() for t in vc]
    return fsx_oracle.expert_tick(w, k, v, np.array([0, rows]), frames.double().cpu().numpy(), EXPERT.n_heads,
                                  EXPERT.head_dim, EXPERT.n_waypoints)[0]


@pytest.mark.parametrize("concurrent", [False, True])
def test_ticks_read_exactly_their_snapshot_while_appends_run(concurrent):
    w, bw, kc, vc, ex, ap, ses, frames = _setup(concurrent)
    try:
        before = [t.clone() for t in kc]
        before_v = [t.clone() for t in vc]
        xs = [synth.make_append_tokens(BACKBONE, 1, 20 + i).cuda() for i in range(3)]
        hidden = [torch.empty(1, BACKBONE.n_new, BACKBONE.d_model, device="cuda") for _ in xs]
        outs, snaps = [], []
        # 12 ticks, an append issued before every fourth one (K = 4), no waiting in between
        for i in range(12):
            if i % 4 == 0:
                ses.append(xs[i // 4], hidden[i // 4])
            out = torch.empty(1, EXPERT.n_waypoints, 2, device="cuda")
            snaps.append(ses.tick(frames, out))
            outs.append(out)
        ses.sync()
        assert ex.status() == fsx.FSX_OK and ap.status() == fsx.FSX_OK
        assert ses.committed() == ses.reserved() == L0 + 3 * BACKBONE.n_new
        # snapshots only grow, in whole appends, and the serial schedule always reads
        # everything reserved before the tick
        assert all(s >= L0 and (s - L0) % BACKBONE.n_new == 0 for s in snaps)
        assert snaps == sorted(snaps)
        if not concurrent:
            assert snaps == [L0 + BACKBONE.n_new * (i // 4 + 1) for i in range(12)]
        for out, s in zip(outs, snaps):
            ref = _oracle_tick(w, kc, vc, s, frames)
            got = out.cpu().double().numpy()[0]
            assert np.linalg.norm(got - ref) <= fc.WAYPOINT_TOL * np.linalg.norm(ref), s
        # the appended rows are the append oracle's, one call after the other
        kn = [t[:L0].float().cpu().numpy() for t in before]
        vn = [t[:L0].float().cpu().numpy() for t in before_v]
        for i, x in enumerate(xs):
            L = L0 + BACKBONE.n_new * i
            _, kr, vr = append_oracle.backbone_append(bw, kn, vn, np.array([0, L]), x.float().cpu().numpy(),
                                                      BACKBONE.n_heads, BACKBONE.head_dim)
            n = BACKBONE.n_new
            for layer in range(BACKBONE.n_layers):
                got_k = kc[layer][L:L + n].float().cpu().numpy()
                got_v = vc[layer][L:L + n].float().cpu().numpy()
                for got, ref in ((got_k, kr[layer]), (got_v, vr[layer])):
                    g2, r2 = got.reshape(n, -1), np.asarray(ref).reshape(n, -1)
                    err = np.max(np.max(np.abs(g2 - r2), axis=-1) / np.max(np.abs(r2), axis=-1))
                    assert err <= 2e-2, (i, layer, err)
                kn[layer] = np.concatenate([kn[layer], got_k])
                vn[layer] = np.concatenate([vn[layer], got_v])
        end = L0 + 3 * BACKBONE.n_new
        for a, b in zip(kc + vc, before + before_v):
            assert torch.equal(a[:L0], b[:L0]) and torch.equal(a[end:], b[end:])
    finally:
        ses.close()
        ap.close()
        ex.close()


def test_append_past_the_capacity_is_refused():
    w, bw, kc, vc, ex, ap, ses, frames = _setup(True)
    try:
        x = synth.make_append_tokens(BACKBONE, 1, 3).cuda()
        hidden = torch.empty(1, BACKBONE.n_new, BACKBONE.d_model, device="cuda")
        for _ in range((CAP - L0) // BACKBONE.n_new):
            ses.append(x, hidden)
        with pytest.raises(fsx.FsxError) as e:
            ses.append(x, hidden)
        assert e.value.status == fsx.FSX_ERR_INVALID_ARG
        ses.sync()
        assert ses.committed() == L0 + BACKBONE.n_new * ((CAP - L0) // BACKBONE.n_new)
    finally:
        ses.close()
        ap.close()
        ex.close()
