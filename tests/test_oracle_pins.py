"""Pins of the fp64 oracle against sources other than itself (CPU only).

Each pin is a function of the oracle module, so the same pins also run against
deliberately broken copies of the oracle (``test_planted_mistake``) to show that
a plausible slip in the oracle -- a dropped term, a wrong axis, a swapped or
transposed operand -- fails at least one of them.

Sources used: torch library routines in float64 (scaled_dot_product_attention,
rms_norm, silu, linear, logsumexp), closed forms of the softmax and of RMSNorm,
the hand-derived cases in tests/golden/, and the invariants the method fixes (Sec. 3.1, Eq. 1: one softmax over the
concatenated keys; backbone cache read-only; vehicles independent).
"""
from __future__ import annotations

import math
import os
import types

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle
from oracle import fsx_oracle
from test_golden import golden_eq1_three_keys, golden_tick_swiglu_closed_form, golden_tick_uniform_attention

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
TINY = dict(n_layers=2, d_model=16, n_heads=2, head_dim=8, d_ff=24,
            n_action=3, n_frame=2, n_waypoints=2)


def _rng(seed):
    return np.random.default_rng(seed)


def tiny_problem(seed=0, lengths=(5, 0, 7), positive=False):
    """Small fp64 problem: weights dict, caches, offsets, frames."""
    r = _rng(seed)
    t = TINY
    nl, d, hd, f = t["n_layers"], t["d_model"], t["n_heads"] * t["head_dim"], t["d_ff"]
    n_tok = t["n_action"] + t["n_frame"]
    p = {
        "act_emb": r.normal(0, 0.5, (t["n_action"], d)),
        "pos_emb": r.normal(0, 0.5, (n_tok, d)),
        "attn_norm": 1 + 0.3 * r.normal(size=(nl, d)),
        "wq": r.normal(0, 1 / math.sqrt(d), (nl, hd, d)),
        "wk": r.normal(0, 1 / math.sqrt(d), (nl, hd, d)),
        "wv": r.normal(0, 1 / math.sqrt(d), (nl, hd, d)),
        "wo": r.normal(0, 1 / math.sqrt(hd), (nl, d, hd)),
        "mlp_norm": 1 + 0.3 * r.normal(size=(nl, d)),
        "w_gate": r.normal(0, 1 / math.sqrt(d), (nl, f, d)),
        "w_up": r.normal(0, 1 / math.sqrt(d), (nl, f, d)),
        "w_down": r.normal(0, 1 / math.sqrt(f), (nl, d, f)),
        "final_norm": 1 + 0.3 * r.normal(size=(d,)),
        "head_w": r.normal(0, 1 / math.sqrt(d), (2, d)),
        "head_b": r.normal(0, 0.5, (2,)),
    }
    offsets = np.concatenate([[0], np.cumsum(lengths)]).astype(np.int64)
    total = int(offsets[-1])
    kc = [r.normal(size=(total, t["n_heads"], t["head_dim"])) * np.exp(0.5 * r.normal(size=(t["n_heads"], t["head_dim"])))
          for _ in range(nl)]
    vc = [r.normal(size=(total, t["n_heads"], t["head_dim"])) for _ in range(nl)]
    frames = r.normal(size=(len(lengths), t["n_frame"], d))
    if positive:
        p["act_emb"] = np.abs(p["act_emb"]) + 0.1
        p["pos_emb"] = np.abs(p["pos_emb"])
        frames = np.abs(frames) + 0.1
        p["mlp_norm"] = np.abs(p["mlp_norm"]) + 0.1
    return p, kc, vc, offsets, frames


def run_tick(orc, p, kc, vc, offsets, frames, capture=False):
    return orc.expert_tick(p, kc, vc, offsets, frames, n_heads=TINY["n_heads"],
                           head_dim=TINY["head_dim"], n_waypoints=TINY["n_waypoints"],
                           capture_attention=capture)


def t64(a):
    return torch.as_tensor(np.asarray(a, dtype=np.float64))


def torch_x0(p, frames):
    """Token assembly through torch ops: [act_emb ; frames] + pos_emb."""
    b = frames.shape[0]
    act = t64(p["act_emb"]).unsqueeze(0).expand(b, -1, -1)
    return torch.cat([act, t64(frames)], dim=1) + t64(p["pos_emb"])


def torch_head(p, x):
    """Waypoint head via torch library routines: Linear(RMSNorm(x))."""
    n = F.rms_norm(x[:, :TINY["n_waypoints"]], (x.shape[-1],), weight=t64(p["final_norm"]), eps=1e-6)
    return F.linear(n, t64(p["head_w"]), t64(p["head_b"])).numpy()


# --------------------------------------------------------------------------- pins
def pin_rms_norm_library(orc):
    """RMSNorm equals torch.nn.functional.rms_norm (eps 1e-6) in fp64."""
    r = _rng(1)
    x = r.normal(size=(7, 33)) * 3
    g = r.normal(size=33)
    ref = F.rms_norm(t64(x), (33,), weight=t64(g), eps=1e-6).numpy()
    np.testing.assert_allclose(orc.rms_norm(x, g), ref, rtol=1e-13, atol=1e-13)


def pin_rms_norm_closed_form(orc):
    """A constant row c normalises to gamma * c / sqrt(c^2 + eps); zero row -> 0."""
    g = np.linspace(-2, 3, 8)
    for c in (2.5, -0.75, 1e-4):
        out = orc.rms_norm(np.full((1, 8), c), g)
        np.testing.assert_allclose(out[0], g * c / math.sqrt(c * c + 1e-6), rtol=1e-14, atol=0)
    assert np.all(orc.rms_norm(np.zeros((2, 8)), g) == 0)


def pin_silu_library(orc):
    """silu equals torch.nn.functional.silu; silu(0)=0, silu(z)->z for large z."""
    z = np.linspace(-30, 30, 401)
    np.testing.assert_allclose(orc.silu(z), F.silu(t64(z)).numpy(), rtol=1e-14, atol=1e-300)
    assert orc.silu(np.array([0.0]))[0] == 0.0
    assert abs(orc.silu(np.array([40.0]))[0] - 40.0) < 1e-12


def _sdpa(q, kc, vc, ko, vo):
    """torch scaled_dot_product_attention over the concatenated keys (Eq. 1)."""
    k = torch.cat([t64(kc), t64(ko)], 0)
    v = torch.cat([t64(vc), t64(vo)], 0)
    out = F.scaled_dot_product_attention(t64(q).transpose(0, 1), k.transpose(0, 1), v.transpose(0, 1))
    return out.transpose(0, 1).numpy()


def pin_attention_library(orc):
    """Eq. 1 equals torch SDPA over [K_vlm; K_ae], [V_vlm; V_ae], incl. an empty cache."""
    r = _rng(2)
    for L, tq, tk in ((9, 4, 4), (0, 5, 5), (1, 3, 6), (40, 7, 2)):
        q = r.normal(size=(tq, 3, 16)) * 2
        kc, vc = r.normal(size=(L, 3, 16)), r.normal(size=(L, 3, 16))
        ko, vo = r.normal(size=(tk, 3, 16)), r.normal(size=(tk, 3, 16))
        np.testing.assert_allclose(orc.attention_eq1(q, kc, vc, ko, vo), _sdpa(q, kc, vc, ko, vo),
                                   rtol=1e-12, atol=1e-12)


def pin_attention_lse_library(orc):
    """The returned log-sum-exp equals torch.logsumexp of the scaled scores."""
    r = _rng(3)
    q, kc, ko = r.normal(size=(4, 2, 8)), r.normal(size=(6, 2, 8)), r.normal(size=(3, 2, 8))
    vc, vo = r.normal(size=(6, 2, 8)), r.normal(size=(3, 2, 8))
    _, lse = orc.attention_eq1(q, kc, vc, ko, vo, return_lse=True)
    k = torch.cat([t64(kc), t64(ko)], 0)
    s = torch.einsum("qhd,khd->hqk", t64(q), k) / math.sqrt(8)
    np.testing.assert_allclose(lse, torch.logsumexp(s, dim=-1).numpy(), rtol=1e-13, atol=1e-13)


def pin_attention_closed_forms(orc):
    """q = 0 or identical keys -> uniform weights -> mean of all values;
    a single key -> that key's value; constant values c -> c."""
    r = _rng(4)
    kc, vc = r.normal(size=(5, 2, 8)), r.normal(size=(5, 2, 8))
    ko, vo = r.normal(size=(3, 2, 8)), r.normal(size=(3, 2, 8))
    v_all = np.concatenate([vc, vo], 0)
    out = orc.attention_eq1(np.zeros((4, 2, 8)), kc, vc, ko, vo)
    np.testing.assert_allclose(out, np.broadcast_to(v_all.mean(0), out.shape), rtol=1e-13, atol=1e-14)
    same = np.broadcast_to(r.normal(size=(1, 2, 8)), (5, 2, 8))
    out = orc.attention_eq1(r.normal(size=(4, 2, 8)), same, vc, same[:3], vo)
    np.testing.assert_allclose(out, np.broadcast_to(v_all.mean(0), out.shape), rtol=1e-13, atol=1e-14)
    out = orc.attention_eq1(r.normal(size=(3, 2, 8)), kc[:0], vc[:0], ko[:1], vo[:1])
    np.testing.assert_allclose(out, np.broadcast_to(vo[0], out.shape), rtol=1e-14, atol=1e-15)
    c = np.full((5, 2, 8), 0.3)
    out = orc.attention_eq1(r.normal(size=(4, 2, 8)) * 5, kc, c, ko, c[:3])
    np.testing.assert_allclose(out, 0.3, rtol=1e-13)


def pin_attention_invariants(orc):
    """Softmax rows sum to 1; permuting cache tokens (K with V) leaves A unchanged;
    duplicating every key/value pair of [cache ; own] leaves A unchanged."""
    r = _rng(5)
    q = r.normal(size=(6, 2, 8)) * 2
    kc, vc = r.normal(size=(11, 2, 8)), r.normal(size=(11, 2, 8))
    ko, vo = r.normal(size=(6, 2, 8)), r.normal(size=(6, 2, 8))
    np.testing.assert_allclose(orc.softmax_row_sums(q, kc, ko), 1.0, rtol=0, atol=1e-12)
    base = orc.attention_eq1(q, kc, vc, ko, vo)
    perm = r.permutation(11)
    np.testing.assert_allclose(orc.attention_eq1(q, kc[perm], vc[perm], ko, vo), base, rtol=1e-12, atol=1e-13)
    dup = orc.attention_eq1(q, np.concatenate([kc, kc]), np.concatenate([vc, vc]),
                            np.concatenate([ko, ko]), np.concatenate([vo, vo]))
    np.testing.assert_allclose(dup, base, rtol=1e-12, atol=1e-13)
    # duplicating only the cache is NOT an invariant (sanity of the test itself)
    half = orc.attention_eq1(q, np.concatenate([kc, kc]), np.concatenate([vc, vc]), ko, vo)
    assert np.max(np.abs(half - base)) > 1e-6


def pin_tick_library_composition(orc):
    """Whole tick equals a composition of torch library routines (rms_norm,
    linear, scaled_dot_product_attention, silu) on a tiny ragged batch."""
    p, kc, vc, offsets, frames = tiny_problem(6)
    got, att = run_tick(orc, p, kc, vc, offsets, frames, capture=True)
    h, dh = TINY["n_heads"], TINY["head_dim"]
    x = torch_x0(p, frames)
    n_tok = x.shape[1]
    for layer in range(TINY["n_layers"]):
        lw = {k: t64(v[layer]) for k, v in p.items() if np.ndim(v) == 3 or k in ("attn_norm", "mlp_norm")}
        for b in range(frames.shape[0]):
            xb = x[b]
            n = F.rms_norm(xb, (xb.shape[-1],), weight=lw["attn_norm"], eps=1e-6)
            q = F.linear(n, lw["wq"]).view(n_tok, h, dh)
            k = F.linear(n, lw["wk"]).view(n_tok, h, dh)
            v = F.linear(n, lw["wv"]).view(n_tok, h, dh)
            lo, hi = offsets[b], offsets[b + 1]
            a = torch.as_tensor(_sdpa(q.numpy(), kc[layer][lo:hi], vc[layer][lo:hi], k.numpy(), v.numpy()))
            a = a.reshape(n_tok, h * dh)
            np.testing.assert_allclose(att[layer, b * n_tok:(b + 1) * n_tok], a.numpy(), rtol=1e-10, atol=1e-12)
            xb = xb + F.linear(a, lw["wo"])
            n = F.rms_norm(xb, (xb.shape[-1],), weight=lw["mlp_norm"], eps=1e-6)
            xb = xb + F.linear(F.silu(F.linear(n, lw["w_gate"])) * F.linear(n, lw["w_up"]), lw["w_down"])
            x[b] = xb
    np.testing.assert_allclose(got, torch_head(p, x), rtol=1e-10, atol=1e-12)


def pin_tick_zero_branches(orc):
    """W_o = W_d = 0 at every layer: the residual stream stays X_0, so the
    waypoints are head(RMSNorm(X_0)) (closed form)."""
    p, kc, vc, offsets, frames = tiny_problem(7)
    p["wo"] = np.zeros_like(p["wo"])
    p["w_down"] = np.zeros_like(p["w_down"])
    got = run_tick(orc, p, kc, vc, offsets, frames)
    np.testing.assert_allclose(got, torch_head(p, torch_x0(p, frames)), rtol=1e-12, atol=1e-13)


def pin_tick_zero_gains(orc):
    """Both norm gains 0: queries, own keys and own values vanish, the softmax is
    uniform over L_b + T keys, the SwiGLU branch is silu(0)*0 = 0, so every token
    of vehicle b gains sum_l (sum of cache V_l rows / (L_b + T)) W_o^l^T."""
    p, kc, vc, offsets, frames = tiny_problem(8)
    p["attn_norm"] = np.zeros_like(p["attn_norm"])
    p["mlp_norm"] = np.zeros_like(p["mlp_norm"])
    got = run_tick(orc, p, kc, vc, offsets, frames)
    x = torch_x0(p, frames)
    n_tok = x.shape[1]
    for b in range(frames.shape[0]):
        lo, hi = offsets[b], offsets[b + 1]
        for layer in range(TINY["n_layers"]):
            mean_v = vc[layer][lo:hi].reshape(hi - lo, TINY["n_heads"] * TINY["head_dim"]).sum(0) / ((hi - lo) + n_tok)
            x[b] = x[b] + torch.as_tensor(p["wo"][layer] @ mean_v)
    np.testing.assert_allclose(got, torch_head(p, x), rtol=1e-12, atol=1e-13)


def pin_tick_uniform_queries(orc):
    """W_q = 0: every query gets uniform weights, so at layer 0 each token's
    attention output is the mean over the cache values and the own values
    V_ae = RMSNorm(X_0) W_v^T (torch routines), and at every layer all tokens of
    a vehicle share one attention row."""
    p, kc, vc, offsets, frames = tiny_problem(9)
    p["wq"] = np.zeros_like(p["wq"])
    _, att = run_tick(orc, p, kc, vc, offsets, frames, capture=True)
    x0 = torch_x0(p, frames)
    n_tok = x0.shape[1]
    for b in range(frames.shape[0]):
        lo, hi = offsets[b], offsets[b + 1]
        n = F.rms_norm(x0[b], (x0.shape[-1],), weight=t64(p["attn_norm"][0]), eps=1e-6)
        v_own = F.linear(n, t64(p["wv"][0])).numpy()
        v_all = np.concatenate([vc[0][lo:hi].reshape(hi - lo, TINY["n_heads"] * TINY["head_dim"]), v_own], 0)
        rows = att[0, b * n_tok:(b + 1) * n_tok]
        np.testing.assert_allclose(rows, np.broadcast_to(v_all.mean(0), rows.shape), rtol=1e-12, atol=1e-13)
        for layer in range(TINY["n_layers"]):
            rows = att[layer, b * n_tok:(b + 1) * n_tok]
            np.testing.assert_allclose(rows, np.broadcast_to(rows[0], rows.shape), rtol=1e-12, atol=1e-13)


def pin_tick_closed_gate(orc):
    """A gate driven to -infinity closes the SwiGLU branch (silu(z) -> 0): with
    positive activations, positive gains, W_gate = -1e4 and W_o = 0 the
    waypoints are head(RMSNorm(X_0))."""
    p, kc, vc, offsets, frames = tiny_problem(10, positive=True)
    p["wo"] = np.zeros_like(p["wo"])
    p["w_gate"] = np.full_like(p["w_gate"], -1e4)
    with np.errstate(over="ignore"):
        got = run_tick(orc, p, kc, vc, offsets, frames)
    np.testing.assert_allclose(got, torch_head(p, torch_x0(p, frames)), rtol=1e-12, atol=1e-13)


def pin_tick_vehicle_independence_and_readonly(orc):
    """Vehicles are independent (changing vehicle 1's cache rows leaves the
    others unchanged) and the tick never writes the cache (Sec. 3.1)."""
    p, kc, vc, offsets, frames = tiny_problem(11)
    kc_before = [k.copy() for k in kc]
    vc_before = [v.copy() for v in vc]
    base = run_tick(orc, p, kc, vc, offsets, frames)
    for a, b in zip(kc + vc, kc_before + vc_before):
        assert np.array_equal(a, b)
    kc2 = [k.copy() for k in kc]
    lo, hi = offsets[2], offsets[3]
    for k in kc2:
        k[lo:hi] = k[lo:hi] * -1.7 + 0.3
    moved = run_tick(orc, p, kc2, vc, offsets, frames)
    np.testing.assert_array_equal(moved[:2], base[:2])
    assert np.max(np.abs(moved[2] - base[2])) > 1e-6


def pin_tick_layer_matching(orc):
    """Expert layer l reads backbone layer l (the layers are matched one to one):
    swapping the two cache layers changes the output, swapping them together
    with the expert layers' weights does not."""
    p, kc, vc, offsets, frames = tiny_problem(12)
    base = run_tick(orc, p, kc, vc, offsets, frames)
    sw = run_tick(orc, p, kc[::-1], vc[::-1], offsets, frames)
    assert np.max(np.abs(sw - base)) > 1e-6
    # with identical expert layers, swapping cache layers together with nothing
    # else must matter; with identical cache layers it must not
    kc_same = [kc[0], kc[0]]
    vc_same = [vc[0], vc[0]]
    a = run_tick(orc, p, kc_same, vc_same, offsets, frames)
    b = run_tick(orc, p, kc_same[::-1], vc_same[::-1], offsets, frames)
    np.testing.assert_array_equal(a, b)


def pin_tick_first_layer_attention(orc):
    """Layer 0's input is the closed-form X_0, so its Eq. 1 output must equal
    torch SDPA of RMSNorm(X_0) projections against backbone cache layer 0."""
    p, kc, vc, offsets, frames = tiny_problem(13)
    _, att = run_tick(orc, p, kc, vc, offsets, frames, capture=True)
    x0 = torch_x0(p, frames)
    n_tok, h, dh = x0.shape[1], TINY["n_heads"], TINY["head_dim"]
    for b in range(frames.shape[0]):
        lo, hi = offsets[b], offsets[b + 1]
        n = F.rms_norm(x0[b], (x0.shape[-1],), weight=t64(p["attn_norm"][0]), eps=1e-6)
        q, k, v = (F.linear(n, t64(p[w][0])).view(n_tok, h, dh).numpy() for w in ("wq", "wk", "wv"))
        ref = _sdpa(q, kc[0][lo:hi], vc[0][lo:hi], k, v).reshape(n_tok, h * dh)
        np.testing.assert_allclose(att[0, b * n_tok:(b + 1) * n_tok], ref, rtol=1e-11, atol=1e-12)


PINS = [pin_rms_norm_library, pin_rms_norm_closed_form, pin_silu_library,
        pin_attention_library, pin_attention_lse_library, pin_attention_closed_forms,
        pin_attention_invariants, pin_tick_library_composition, pin_tick_zero_branches,
        pin_tick_zero_gains, pin_tick_uniform_queries, pin_tick_closed_gate,
        pin_tick_vehicle_independence_and_readonly, pin_tick_layer_matching,
        pin_tick_first_layer_attention, golden_eq1_three_keys, golden_tick_uniform_attention,
        golden_tick_swiglu_closed_form]


@pytest.mark.parametrize("pin", PINS, ids=lambda f: f.__name__)
def test_pin(pin):
    pin(oracle)


# ---------------------------------------------------------------- planted mistakes
MUTATIONS = {
    "no_score_scale": ("scale = 1.0 / np.sqrt(d)", "scale = 1.0"),
    "softmax_wrong_axis": ("z = np.sum(e, axis=1, keepdims=True)", "z = np.sum(e, axis=0, keepdims=True)"),
    "lse_missing_max": ("lse[h, :] = (m + np.log(z))[:, 0]", "lse[h, :] = np.log(z)[:, 0]"),
    "cache_keys_dropped": ("kc[lo:hi]", "kc[lo:lo]"),
    "cache_values_dropped": ("vc[lo:hi]", "vc[lo:lo]"),
    "own_keys_dropped": ("attention_eq1(q_ae, k_vlm, v_vlm, k_ae, v_ae)",
                         "attention_eq1(q_ae, k_vlm, v_vlm, k_ae[:0], v_ae[:0])"),
    "keys_as_queries": ("a = attention_eq1(q_ae, k_vlm", "a = attention_eq1(k_ae, k_vlm"),
    "wo_transposed_layout": ("a @ wo.T", "a @ wo.reshape(wo.shape[1], wo.shape[0])"),
    "attn_residual_dropped": ("x[b] = x[b] + a @ wo.T", "x[b] = a @ wo.T"),
    "mlp_residual_dropped": ("x[b] = x[b] + (silu(", "x[b] = (silu("),
    "gate_up_swapped": ("silu(n @ wg.T) * (n @ wu.T)", "silu(n @ wu.T) * (n @ wg.T)"),
    "silu_is_sigmoid": ("return z / (1.0 + np.exp(-z))", "return 1.0 / (1.0 + np.exp(-z))"),
    "rms_gamma_dropped": ("np.sqrt(ms + eps) * np.asarray(gamma, dtype=np.float64)", "np.sqrt(ms + eps)"),
    "rms_eps_outside": ("np.sqrt(ms + eps)", "(np.sqrt(ms) + eps)"),
    "rms_sum_not_mean": ("np.mean(x * x, axis=-1", "np.sum(x * x, axis=-1"),
    "pos_emb_dropped": ("x = x + pos_emb[None, :, :]", "x = x"),
    "head_bias_dropped": ("@ head_w.T + head_b", "@ head_w.T"),
    "final_norm_dropped": ("rms_norm(x[:, :n_waypoints, :], final_norm)", "x[:, :n_waypoints, :]"),
    "waypoints_from_frames": ("x[:, :n_waypoints, :]", "x[:, -n_waypoints:, :]"),
    "cache_layer_off_by_one": ("kc = k_cache[layer]", "kc = k_cache[layer - 1]"),
    "norm_gains_swapped": ('g1 = _layer(params, layer, "attn_norm")', 'g1 = _layer(params, layer, "mlp_norm")'),
    "wk_wv_swapped": ('wk = _layer(params, layer, "wk")', 'wk = _layer(params, layer, "wv")'),
}


def _mutant(name):
    src_path = fsx_oracle.__file__
    with open(src_path) as fh:
        src = fh.read()
    old, new = MUTATIONS[name]
    assert src.count(old) >= 1, f"mutation {name!r} no longer matches the oracle source"
    mod = types.ModuleType(f"oracle_mutant_{name}")
    mod.__file__ = src_path
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
