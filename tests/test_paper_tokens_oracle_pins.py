"""Pins of the fp64 oracle of the paper's ten-token expert layout (CPU only).

Sources other than the oracle: a composition of torch routines in float64 (linear, silu,
rms_norm, scaled_dot_product_attention), closed forms with the attention and SwiGLU
branches zeroed, and invariants of the layout (Sec. 3.1: the state token carries the ego
state into every layer; the head decodes the five query tokens). ``test_planted_mistake``
runs every pin against deliberately broken copies of the oracle.
"""
from __future__ import annotations

import math
import types

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle import paper_tokens_oracle
from test_oracle_pins import TINY, _sdpa, t64, tiny_problem

N_TOK = 1 + paper_tokens_oracle.N_VISUAL + paper_tokens_oracle.N_QUERY


def paper_problem(seed=0, lengths=(5, 0, 7)):
    p, kc, vc, offsets, _ = tiny_problem(seed, lengths)
    r = np.random.default_rng(seed + 100)
    d = TINY["d_model"]
    p.update({
        "state_w1": r.normal(0, 1 / math.sqrt(16), (d, 16)),
        "state_b1": r.normal(0, 0.3, d),
        "state_w2": r.normal(0, 1 / math.sqrt(d), (d, d)),
        "state_b2": r.normal(0, 0.3, d),
        "query_emb": r.normal(0, 0.5, (5, d)),
        "pos_emb": r.normal(0, 0.5, (N_TOK, d)),
        "head_w1": r.normal(0, 1 / math.sqrt(d), (d, d)),
        "head_b1": r.normal(0, 0.3, d),
        "head_w2": r.normal(0, 1 / math.sqrt(d), (2, d)),
        "head_b2": r.normal(0, 0.3, 2),
    })
    B = len(lengths)
    visual = r.normal(size=(B, 4, d))
    state = r.normal(size=(B, 16))
    return p, kc, vc, offsets, visual, state


def run(orc, p, kc, vc, offsets, visual, state):
    return orc.expert_tick_paper_tokens(p, kc, vc, offsets, visual, state, TINY["n_heads"], TINY["head_dim"])


def torch_tokens(p, visual, state):
    """[state MLP(s) ; visual ; queries] + positions, through torch routines."""
    s = F.linear(F.silu(F.linear(t64(state), t64(p["state_w1"]), t64(p["state_b1"]))), t64(p["state_w2"]),
                 t64(p["state_b2"]))
    q = t64(p["query_emb"]).unsqueeze(0).expand(visual.shape[0], -1, -1)
    return torch.cat([s.unsqueeze(1), t64(visual), q], dim=1) + t64(p["pos_emb"])


def torch_head(p, x):
    n = F.rms_norm(x[:, 5:], (x.shape[-1],), weight=t64(p["final_norm"]), eps=1e-6)
    h = F.silu(F.linear(n, t64(p["head_w1"]), t64(p["head_b1"])))
    return F.linear(h, t64(p["head_w2"]), t64(p["head_b2"])).numpy()


# ---------------------------------------------------------------- pins
def pin_library_composition(orc):
    """The whole ten-token tick equals a composition of torch routines."""
    p, kc, vc, offsets, visual, state = paper_problem(1)
    got = run(orc, p, kc, vc, offsets, visual, state)
    h, dh = TINY["n_heads"], TINY["head_dim"]
    x = torch_tokens(p, visual, state)
    for layer in range(TINY["n_layers"]):
        lw = {k: t64(p[k][layer]) for k in ("attn_norm", "wq", "wk", "wv", "wo", "mlp_norm", "w_gate", "w_up",
                                             "w_down")}
        for b in range(visual.shape[0]):
            xb = x[b]
            n = F.rms_norm(xb, (xb.shape[-1],), weight=lw["attn_norm"], eps=1e-6)
            q = F.linear(n, lw["wq"]).view(N_TOK, h, dh)
            k = F.linear(n, lw["wk"]).view(N_TOK, h, dh)
            v = F.linear(n, lw["wv"]).view(N_TOK, h, dh)
            lo, hi = offsets[b], offsets[b + 1]
            a = torch.as_tensor(_sdpa(q.numpy(), kc[layer][lo:hi], vc[layer][lo:hi], k.numpy(), v.numpy()))
            xb = xb + F.linear(a.reshape(N_TOK, h * dh), lw["wo"])
            n = F.rms_norm(xb, (xb.shape[-1],), weight=lw["mlp_norm"], eps=1e-6)
            xb = xb + F.linear(F.silu(F.linear(n, lw["w_gate"])) * F.linear(n, lw["w_up"]), lw["w_down"])
            x[b] = xb
    np.testing.assert_allclose(got, torch_head(p, x), rtol=1e-10, atol=1e-12)


def pin_zero_branches(orc):
    """W_o = W_d = 0 at every layer: each query token keeps its input, so every vehicle's
    waypoints equal the head of (query embedding + position), whatever the state, the
    visual tokens and the cache."""
    p, kc, vc, offsets, visual, state = paper_problem(2)
    p["wo"] = np.zeros_like(p["wo"])
    p["w_down"] = np.zeros_like(p["w_down"])
    got = run(orc, p, kc, vc, offsets, visual, state)
    q = (t64(p["query_emb"]) + t64(p["pos_emb"][5:])).unsqueeze(0)
    n = F.rms_norm(q, (q.shape[-1],), weight=t64(p["final_norm"]), eps=1e-6)
    want = F.linear(F.silu(F.linear(n, t64(p["head_w1"]), t64(p["head_b1"]))), t64(p["head_w2"]),
                    t64(p["head_b2"])).numpy()[0]
    for b in range(visual.shape[0]):
        np.testing.assert_allclose(got[b], want, rtol=1e-12, atol=1e-13)


def pin_state_reaches_the_waypoints(orc):
    """The state token feeds every layer through attention: changing the ego state changes
    every waypoint; with W_s1 = 0 the state token is a constant and the state no longer matters."""
    p, kc, vc, offsets, visual, state = paper_problem(3)
    base = run(orc, p, kc, vc, offsets, visual, state)
    moved = run(orc, p, kc, vc, offsets, visual, state + 1.0)
    assert np.min(np.abs(moved - base)) > 0
    p["state_w1"] = np.zeros_like(p["state_w1"])
    a = run(orc, p, kc, vc, offsets, visual, state)
    b = run(orc, p, kc, vc, offsets, visual, state * -3.0)
    np.testing.assert_array_equal(a, b)


def pin_vehicle_independence(orc):
    """A vehicle's waypoints depend only on its own state, visual tokens and cache rows."""
    p, kc, vc, offsets, visual, state = paper_problem(4)
    base = run(orc, p, kc, vc, offsets, visual, state)
    v2, s2 = visual.copy(), state.copy()
    v2[1] += 0.7
    s2[1] -= 0.4
    kc2 = [k.copy() for k in kc]
    for k in kc2:
        k[offsets[2]:offsets[3]] *= -1.0
    got = run(orc, p, kc2, vc, offsets, v2, s2)
    np.testing.assert_array_equal(got[0], base[0])
    assert np.max(np.abs(got[1] - base[1])) > 1e-9 and np.max(np.abs(got[2] - base[2])) > 1e-9


PINS = [pin_library_composition, pin_zero_branches, pin_state_reaches_the_waypoints, pin_vehicle_independence]


@pytest.mark.parametrize("pin", PINS, ids=lambda f: f.__name__)
def test_pin(pin):
    pin(paper_tokens_oracle)


# ---------------------------------------------------------------- planted mistakes
MUTATIONS = {
    "head_on_first_tokens": ("x[:, 1 + N_VISUAL:, :]", "x[:, :N_QUERY, :]"),
    "head_without_silu": ('h = silu(n @ np.asarray(params["head_w1"], np.float64).T + np.asarray(params["head_b1"], np.float64))',
                          'h = n @ np.asarray(params["head_w1"], np.float64).T + np.asarray(params["head_b1"], np.float64)'),
    "head_without_norm": ('n = rms_norm(q_tokens, np.asarray(params["final_norm"], np.float64))', "n = q_tokens"),
    "state_bias_dropped": (' + np.asarray(params["state_b1"], np.float64))', ")"),
    "positions_dropped": ('x = x + np.asarray(params["pos_emb"], np.float64)[None, :, :]', "x = x"),
    "visual_and_queries_swapped": ("np.concatenate([t_state[:, None, :], visual,\n                        np.broadcast_to(queries, (n_batch,) + queries.shape)], axis=1)",
                                   "np.concatenate([t_state[:, None, :], np.broadcast_to(queries, (n_batch,) + queries.shape)[:, :4],\n                        np.concatenate([visual, visual[:, :1]], axis=1)], axis=1)"),
    "state_token_last": ("np.concatenate([t_state[:, None, :], visual,\n                        np.broadcast_to(queries, (n_batch,) + queries.shape)], axis=1)",
                         "np.concatenate([visual, np.broadcast_to(queries, (n_batch,) + queries.shape),\n                        t_state[:, None, :]], axis=1)"),
}


def _mutant(name):
    src_path = paper_tokens_oracle.__file__
    with open(src_path) as fh:
        src = fh.read()
    old, new = MUTATIONS[name]
    assert src.count(old) >= 1, f"mutation {name!r} no longer matches the oracle source"
    mod = types.ModuleType(f"oracle.paper_tokens_mutant_{name}")
    mod.__file__ = src_path
    mod.__package__ = "oracle"
    exec(compile(src.replace(old, new), src_path, "exec"), mod.__dict__)
    return mod


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_planted_mistake(name):
    mod = _mutant(name)
    caught = []
    for pin in PINS:
        try:
            with np.errstate(all="ignore"):
                pin(mod)
        except Exception:  # AssertionError or a shape error both count
            caught.append(pin.__name__)
    assert caught, f"no pin catches the planted mistake {name!r}"
