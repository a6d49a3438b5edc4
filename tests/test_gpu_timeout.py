"""The bounded-wait timeout path of the single-launch tick, exercised without breaking
any kernel: a test hook lowers the limit of the tick's device-wide counter waits to
1 ns, so the first wait that finds its counter incomplete gives up at once. The tick
must end (every CTA drains what it has in flight: its cache-row copies, the weight
copies it issued, its MMAs, its partners' stores), report FSX_ERR_TIMEOUT and write no
waypoint; with the default limit restored, the next tick on the same handle must match
the oracle."""
from __future__ import annotations

import time

import numpy as np
import pytest
import torch

from paper_2607_15621_gb300 import fsx, synth

import fsx_cases as fc

pytestmark = pytest.mark.gpu


def test_wait_timeout_is_reported_and_the_next_tick_is_clean():
    case = fc.Case(synth.Dims(n_layers=4), [100], "bf16", seed=12)
    ex = case.expert()
    try:
        assert ex.launches(1) == 1  # the single-launch tick
        ex.set_wait_limit(1)
        out = torch.full((1, case.dims.n_waypoints, 2), 123.0, device="cuda")
        t0 = time.perf_counter()
        ex.tick(case.k, case.v, case.offsets, case.frames, out)
        torch.cuda.synchronize()
        elapsed = time.perf_counter() - t0
        assert ex.status() == fsx.FSX_ERR_TIMEOUT
        assert torch.all(out == 123.0)  # no waypoint from a timed-out tick
        assert elapsed < 30.0  # bounded: at most about a second per wait that runs out
        ex.set_wait_limit(0)  # the default limit again
        wp = fc.run_tick(ex, case)
    finally:
        ex.close()
    ref, _ = case.oracle_vehicle(0)
    assert np.linalg.norm(wp[0] - ref[0]) <= fc.WAYPOINT_TOL * np.linalg.norm(ref[0])
