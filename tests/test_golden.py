"""The fp64 oracle against the hand-derived closed forms in tests/golden/ (CPU only).

The paper prints no worked example, so each fixture is a small case whose exact result
follows from Eq. 1 and the layer of Sec. 3.1 by the arithmetic written in the fixture's
`derivation` field."""
from __future__ import annotations

import json
import math
import os

import numpy as np

from oracle import fsx_oracle

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _load(name):
    with open(os.path.join(GOLDEN, name)) as fh:
        return json.load(fh)


def golden_eq1_three_keys(orc):
    """Eq. 1 over two cache keys and one own key against its hand-derived result."""
    g = _load("eq1_three_keys.json")
    q = np.asarray(g["q_over_sqrt2_ln2"]) * math.sqrt(2.0) * math.log(2.0)
    # oracle layout: q [T, H, D], cache [L, H, D], own [T_own, H, D]
    out, lse = orc.attention_eq1(q[None, None, :], np.asarray(g["k_cache"])[:, None, :],
                                        np.asarray(g["v_cache"])[:, None, :], np.asarray(g["k_own"])[:, None, :],
                                        np.asarray(g["v_own"])[:, None, :], return_lse=True)
    np.testing.assert_allclose(out[0, 0], g["output"], rtol=0, atol=1e-12)
    # log-sum-exp of the scores: ln(7/2)
    np.testing.assert_allclose(np.ravel(lse)[0], math.log(3.5), rtol=0, atol=1e-12)
    sums = orc.softmax_row_sums(q[None, None, :], np.asarray(g["k_cache"])[:, None, :],
                                       np.asarray(g["k_own"])[:, None, :])
    np.testing.assert_allclose(np.ravel(sums), 1.0, rtol=0, atol=1e-12)
    w = np.array([a / b for a, b in g["weights"]])
    np.testing.assert_allclose(w.sum(), 1.0, atol=1e-15)
    np.testing.assert_allclose(w @ np.vstack([g["v_cache"], g["v_own"]]), g["output"], atol=1e-12)


def golden_tick_uniform_attention(orc):
    """A one-layer tick with uniform attention against its hand-derived waypoint."""
    g = _load("tick_uniform_attention.json")
    keys = ["act_emb", "pos_emb", "attn_norm", "wq", "wk", "wv", "wo", "mlp_norm", "w_gate", "w_up", "w_down",
            "final_norm", "head_w", "head_b"]
    p = {k: np.asarray(g[k], dtype=np.float64) for k in keys}
    kc = [np.asarray(g["k_cache"], dtype=np.float64)]
    vc = [np.asarray(g["v_cache"], dtype=np.float64)]
    frames = np.asarray(g["frames"], dtype=np.float64)
    wp, att = orc.expert_tick(p, kc, vc, np.array([0, 2]), frames, n_heads=1, head_dim=2, n_waypoints=1,
                                     capture_attention=True)
    num = [a / b for a, b in g["waypoint0_numerators"]]
    ms = g["mean_square_token0"][0] / g["mean_square_token0"][1]
    r = math.sqrt(ms + g["eps"])
    want = [num[0] / r + g["waypoint0_offsets"][0], num[1] / r + g["waypoint0_offsets"][1]]
    np.testing.assert_allclose(np.ravel(wp), want, rtol=0, atol=1e-12)
    np.testing.assert_allclose(np.asarray(att).reshape(-1, 2), np.tile(g["attention_output_every_token"], (2, 1)),
                               rtol=0, atol=1e-12)


def golden_tick_swiglu_closed_form(orc):
    """A one-layer tick whose SwiGLU block is evaluated in closed form (W_o = 0, empty cache)."""
    g = _load("tick_swiglu_closed_form.json")
    keys = ["act_emb", "pos_emb", "attn_norm", "wq", "wk", "wv", "wo", "mlp_norm", "w_up", "w_down",
            "final_norm", "head_w", "head_b"]
    p = {k: np.asarray(g[k], dtype=np.float64) for k in keys}
    ln3 = math.log(3.0)
    p["w_gate"] = np.array([[np.asarray(g["w_gate_row0_over_ln3"]) * ln3, [0.0, 0.0]]])
    empty = [np.zeros((0, 1, 2))]
    frames = np.asarray(g["frames"], dtype=np.float64)
    wp = orc.expert_tick(p, empty, empty, np.array([0, 0]), frames, n_heads=1, head_dim=2, n_waypoints=1)
    eps = g["eps"]
    x0 = g["x0_token0"]
    c = 2.0 / math.sqrt((x0[0] ** 2 + x0[1] ** 2) / 2 + eps)
    z = c * ln3
    h0 = z / (1.0 + math.exp(-z)) * c
    x2 = (x0[0] + h0, x0[1])
    r = math.sqrt((x2[0] ** 2 + x2[1] ** 2) / 2 + eps)
    np.testing.assert_allclose(np.ravel(wp), [x2[0] / r, x2[1] / r], rtol=0, atol=1e-12)


def test_eq1_three_keys():
    golden_eq1_three_keys(fsx_oracle)


def test_tick_uniform_attention():
    golden_tick_uniform_attention(fsx_oracle)


def test_tick_swiglu_closed_form():
    golden_tick_swiglu_closed_form(fsx_oracle)
