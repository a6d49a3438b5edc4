"""Pins of the fp64 oracle of the staleness-masked clip forward (CPU only).

Sources other than the oracle: the per-block attention-mask formulation the paper
trains with (Sec. 3.2: all frames of a clip in one pass, one attention over every
block's tokens with a boolean mask), written with torch routines in float64; closed
values of the visible prefix; and invariants (rows a block cannot see do not matter).
``test_planted_mistake`` runs every pin against deliberately broken copies of the oracle.
"""
from __future__ import annotations

import types

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle import staleness_oracle
from test_oracle_pins import TINY, t64, tiny_problem, torch_head

TEXT, TPF, J = 6, 4, 5   # text rows, rows per frame, frames per clip


def clip_problem(seed=0):
    p, _, _, _, _ = tiny_problem(seed)
    r = np.random.default_rng(seed + 200)
    rows = TEXT + TPF * J
    h, dh = TINY["n_heads"], TINY["head_dim"]
    kc = [r.normal(size=(rows, h, dh)) * 1.5 for _ in range(TINY["n_layers"])]
    vc = [r.normal(size=(rows, h, dh)) for _ in range(TINY["n_layers"])]
    frames = r.normal(size=(J, TINY["n_frame"], TINY["d_model"]))
    return p, kc, vc, frames


def run(orc, p, kc, vc, frames, delta):
    return orc.staleness_masked_forward(p, kc, vc, TEXT, frames, delta, TINY["n_heads"], TINY["head_dim"],
                                        TINY["n_waypoints"], TPF)


def block_mask_forward(p, kc, vc, frames, delta):
    """All blocks of the clip in one pass: one SDPA per layer over [clip cache ; every
    block's own keys] with a boolean mask (block j: its visible cache prefix and its own
    keys only)."""
    h, dh = TINY["n_heads"], TINY["head_dim"]
    n_act = TINY["n_action"]
    T = n_act + TINY["n_frame"]
    rows = kc[0].shape[0]
    act = t64(p["act_emb"]).unsqueeze(0).expand(J, -1, -1)
    x = (torch.cat([act, t64(frames)], dim=1) + t64(p["pos_emb"])).reshape(J * T, -1)
    mask = torch.zeros(J * T, rows + J * T, dtype=torch.bool)
    for j in range(J):
        pj = TEXT if j < delta else TEXT + TPF * (j - delta + 1)
        mask[j * T:(j + 1) * T, :pj] = True
        mask[j * T:(j + 1) * T, rows + j * T:rows + (j + 1) * T] = True
    for layer in range(TINY["n_layers"]):
        g = {k: t64(p[k][layer]) for k in ("attn_norm", "wq", "wk", "wv", "wo", "mlp_norm", "w_gate", "w_up",
                                            "w_down")}
        n = F.rms_norm(x, (x.shape[-1],), weight=g["attn_norm"], eps=1e-6)
        q = F.linear(n, g["wq"]).view(J * T, h, dh)
        k = torch.cat([t64(kc[layer]), F.linear(n, g["wk"]).view(J * T, h, dh)], 0)
        v = torch.cat([t64(vc[layer]), F.linear(n, g["wv"]).view(J * T, h, dh)], 0)
        a = F.scaled_dot_product_attention(q.transpose(0, 1), k.transpose(0, 1), v.transpose(0, 1),
                                           attn_mask=mask).transpose(0, 1).reshape(J * T, h * dh)
        x = x + F.linear(a, g["wo"])
        n = F.rms_norm(x, (x.shape[-1],), weight=g["mlp_norm"], eps=1e-6)
        x = x + F.linear(F.silu(F.linear(n, g["w_gate"])) * F.linear(n, g["w_up"]), g["w_down"])
    return torch_head(p, x.view(J, T, -1))


# ---------------------------------------------------------------- pins
def pin_block_mask_formulation(orc):
    """The clip forward equals the one-pass per-block-mask formulation, for several delta."""
    p, kc, vc, frames = clip_problem(1)
    for delta in (0, 1, 2, 5, 7):
        np.testing.assert_allclose(run(orc, p, kc, vc, frames, delta), block_mask_forward(p, kc, vc, frames, delta),
                                   rtol=1e-10, atol=1e-12)


def pin_visible_prefix_values(orc):
    """Frame j with staleness delta sees the text plus frames 0 .. j - delta (text only if j < delta)."""
    vp = orc.visible_prefix
    assert vp(0, 0, 32) == 36 and vp(3, 0, 32) == 48 and vp(3, 1, 32) == 44
    assert vp(0, 1, 32) == 32 and vp(2, 3, 32) == 32 and vp(3, 3, 32) == 36


def pin_unseen_rows_do_not_matter(orc):
    """With delta = 2 the last two frames' cache rows are seen by no block; frame 0's rows
    reach blocks 2 .. J-1 but not blocks 0 and 1 (which see the text only)."""
    p, kc, vc, frames = clip_problem(2)
    base = run(orc, p, kc, vc, frames, 2)
    kc2 = [k.copy() for k in kc]
    for k in kc2:
        k[TEXT + TPF * (J - 2):] = -3.0 * k[TEXT + TPF * (J - 2):]
    np.testing.assert_array_equal(run(orc, p, kc2, vc, frames, 2), base)
    vc3 = [v.copy() for v in vc]
    for v in vc3:
        v[TEXT:TEXT + TPF] += 2.0
    got = run(orc, p, kc, vc3, frames, 2)
    np.testing.assert_array_equal(got[:2], base[:2])
    assert np.min(np.max(np.abs(got[2:] - base[2:]), axis=(1, 2))) > 1e-9


PINS = [pin_block_mask_formulation, pin_visible_prefix_values, pin_unseen_rows_do_not_matter]


@pytest.mark.parametrize("pin", PINS, ids=lambda f: f.__name__)
def test_pin(pin):
    pin(staleness_oracle)


# ---------------------------------------------------------------- planted mistakes
MUTATIONS = {
    "prefix_excludes_frame_j_minus_delta": ("tokens_per_frame * (j - delta + 1)", "tokens_per_frame * (j - delta)"),
    "text_only_condition_off_by_one": ("if j < delta:", "if j <= delta:"),
    "delta_ignored": ("p_j = visible_prefix(j, delta, text_len, tokens_per_frame)",
                      "p_j = visible_prefix(j, 0, text_len, tokens_per_frame)"),
    "whole_cache_visible": ("kc = [k[:p_j] for k in k_cache]\n        vc = [v[:p_j] for v in v_cache]",
                            "kc = list(k_cache)\n        vc = list(v_cache)\n        p_j = len(kc[0])"),
}


def _mutant(name):
    src_path = staleness_oracle.__file__
    with open(src_path) as fh:
        src = fh.read()
    old, new = MUTATIONS[name]
    assert src.count(old) >= 1, f"mutation {name!r} no longer matches the oracle source"
    mod = types.ModuleType(f"oracle.staleness_mutant_{name}")
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
