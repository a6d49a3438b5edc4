"""Pins of the fp64 oracle of the incremental cache append (CPU only).

Sources other than the oracle itself: torch routines in float64 (RoPE written as
complex multiplication with torch.polar, rms_norm, linear, silu,
scaled_dot_product_attention with a causal or explicit mask), closed forms of the
rotary embedding, and the properties the paper states or the method fixes: the
append is exact against a monolithic forward (Sec. 1, Sec. 3.3: the golden
equivalence of incremental and monolithic prefill), causality, vehicle
independence and a read-only cache. ``test_planted_mistake`` runs every pin
against deliberately broken copies of the oracle.
"""
from __future__ import annotations

import math
import types

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle import append_oracle

TINY = dict(n_layers=2, d_model=16, n_heads=2, head_dim=8, d_ff=24)


def tiny_params(seed=0):
    r = np.random.default_rng(seed)
    nl, d, hd, f = TINY["n_layers"], TINY["d_model"], TINY["n_heads"] * TINY["head_dim"], TINY["d_ff"]
    return {
        "attn_norm": 1 + 0.3 * r.normal(size=(nl, d)),
        "wq": r.normal(0, 1 / math.sqrt(d), (nl, hd, d)) * 2.0,
        "wk": r.normal(0, 1 / math.sqrt(d), (nl, hd, d)) * 2.0,
        "wv": r.normal(0, 1 / math.sqrt(d), (nl, hd, d)),
        "wo": r.normal(0, 1 / math.sqrt(hd), (nl, d, hd)),
        "mlp_norm": 1 + 0.3 * r.normal(size=(nl, d)),
        "w_gate": r.normal(0, 1 / math.sqrt(d), (nl, f, d)),
        "w_up": r.normal(0, 1 / math.sqrt(d), (nl, f, d)),
        "w_down": r.normal(0, 1 / math.sqrt(f), (nl, d, f)),
    }


def tiny_tokens(n, seed=1):
    return np.random.default_rng(seed).normal(size=(n, TINY["d_model"]))


def t64(a):
    return torch.as_tensor(np.asarray(a, dtype=np.float64))


def torch_rope(x, positions, base=append_oracle.ROPE_BASE):
    """RoPE as complex multiplication: (x_j + i x_{j+D/2}) * exp(i pos base^(-2j/D))."""
    x = t64(x)
    d = x.shape[-1]
    inv_freq = 1.0 / (base ** (torch.arange(0, d, 2, dtype=torch.float64) / d))
    ang = torch.outer(t64(positions), inv_freq)                        # [S, D/2]
    rot = torch.polar(torch.ones_like(ang), ang)[:, None, :]           # [S, 1, D/2]
    z = torch.complex(x[..., : d // 2], x[..., d // 2:]) * rot
    return torch.cat([z.real, z.imag], dim=-1)


def torch_layer_stack(p, x, positions, k_prefix=None, v_prefix=None, mask=None):
    """The decoder stack written with torch library routines; returns (h, k rows, v rows)."""
    h_, dh = TINY["n_heads"], TINY["head_dim"]
    x = t64(x)
    s = x.shape[0]
    ks, vs = [], []
    for layer in range(len(p["wq"])):
        n = F.rms_norm(x, (x.shape[-1],), weight=t64(p["attn_norm"][layer]), eps=1e-6)
        q = torch_rope(F.linear(n, t64(p["wq"][layer])).view(s, h_, dh), positions)
        k = torch_rope(F.linear(n, t64(p["wk"][layer])).view(s, h_, dh), positions)
        v = F.linear(n, t64(p["wv"][layer])).view(s, h_, dh)
        ks.append(k)
        vs.append(v)
        if k_prefix is None:
            a = F.scaled_dot_product_attention(q.transpose(0, 1), k.transpose(0, 1), v.transpose(0, 1),
                                               is_causal=True)
        else:
            kk = torch.cat([t64(k_prefix[layer]), k], 0)
            vv = torch.cat([t64(v_prefix[layer]), v], 0)
            a = F.scaled_dot_product_attention(q.transpose(0, 1), kk.transpose(0, 1), vv.transpose(0, 1),
                                               attn_mask=mask)
        x = x + F.linear(a.transpose(0, 1).reshape(s, h_ * dh), t64(p["wo"][layer]))
        n = F.rms_norm(x, (x.shape[-1],), weight=t64(p["mlp_norm"][layer]), eps=1e-6)
        x = x + F.linear(F.silu(F.linear(n, t64(p["w_gate"][layer]))) * F.linear(n, t64(p["w_up"][layer])),
                         t64(p["w_down"][layer]))
    return x.numpy(), torch.stack(ks).numpy(), torch.stack(vs).numpy()


def prefill(orc, p, x):
    return orc.backbone_prefill(p, x, TINY["n_heads"], TINY["head_dim"])


def append(orc, p, kc, vc, offsets, x_new):
    return orc.backbone_append(p, kc, vc, offsets, x_new, TINY["n_heads"], TINY["head_dim"])


# ---------------------------------------------------------------- pins
def pin_rope_complex(orc):
    """RoPE equals complex multiplication by exp(i pos theta_j) of the pairs (j, j + D/2)."""
    x = np.random.default_rng(3).normal(size=(7, 3, 8))
    pos = np.array([0, 1, 2, 5, 17, 100, 4095])
    np.testing.assert_allclose(orc.rope(x, pos), torch_rope(x, pos).numpy(), rtol=1e-13, atol=1e-13)


def pin_rope_closed_forms(orc):
    """Position 0 is the identity; each pair keeps its length; with D = 2 the single pair
    turns by exactly pos radians; scores depend only on the distance of the positions."""
    r = np.random.default_rng(4)
    x = r.normal(size=(5, 2, 8))
    np.testing.assert_allclose(orc.rope(x, np.zeros(5)), x, rtol=0, atol=1e-15)
    y = orc.rope(x, np.array([3, 9, 27, 81, 243]))
    np.testing.assert_allclose(y[..., :4] ** 2 + y[..., 4:] ** 2, x[..., :4] ** 2 + x[..., 4:] ** 2, rtol=1e-12)
    one = np.array([[[1.0, 0.0]], [[0.0, 2.0]]])
    got = orc.rope(one, np.array([1, 3]))
    np.testing.assert_allclose(got[0, 0], [math.cos(1.0), math.sin(1.0)], atol=1e-15)
    np.testing.assert_allclose(got[1, 0], [-2 * math.sin(3.0), 2 * math.cos(3.0)], atol=1e-15)
    q = r.normal(size=(1, 1, 8))
    k = r.normal(size=(1, 1, 8))
    s1 = np.sum(orc.rope(q, [11]) * orc.rope(k, [4]))
    s2 = np.sum(orc.rope(q, [111]) * orc.rope(k, [104]))
    np.testing.assert_allclose(s1, s2, rtol=1e-11)


def pin_prefill_library(orc):
    """The monolithic forward equals the torch composition with causal SDPA."""
    p = tiny_params(5)
    x = tiny_tokens(9, 6)
    h, k, v = prefill(orc, p, x)
    th, tk, tv = torch_layer_stack(p, x, np.arange(9))
    np.testing.assert_allclose(h, th, rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(k, tk, rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(v, tv, rtol=1e-11, atol=1e-12)


def pin_append_library(orc):
    """The append equals the torch composition with an explicit prefix + causal mask."""
    p = tiny_params(7)
    r = np.random.default_rng(8)
    n_cached, n_app = 6, 4
    kc = [r.normal(size=(n_cached, 2, 8)) for _ in range(2)]
    vc = [r.normal(size=(n_cached, 2, 8)) for _ in range(2)]
    x = tiny_tokens(n_app, 9)
    h, k, v = append(orc, p, kc, vc, np.array([0, n_cached]), x[None])
    mask = torch.ones(n_app, n_cached + n_app, dtype=torch.bool)
    mask[:, n_cached:] = torch.tril(torch.ones(n_app, n_app, dtype=torch.bool))
    th, tk, tv = torch_layer_stack(p, x, n_cached + np.arange(n_app), kc, vc, mask)
    np.testing.assert_allclose(h[0], th, rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(k, tk, rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(v, tv, rtol=1e-11, atol=1e-12)


def pin_incremental_equals_monolithic(orc):
    """The paper's golden equivalence (Sec. 1, Sec. 3.3): appending A tokens to the cache
    of a prefix gives the rows and hidden states of the monolithic forward over the whole
    sequence, for any prefix length, also one token at a time."""
    p = tiny_params(10)
    x = tiny_tokens(13, 11)
    n_app = 4
    for n_cached in (0, 1, 5, 9):
        h_full, k_full, v_full = prefill(orc, p, x[:n_cached + n_app])
        _, kc, vc = prefill(orc, p, x[:n_cached])
        h, k, v = append(orc, p, list(kc), list(vc), np.array([0, n_cached]), x[None, n_cached:n_cached + n_app])
        np.testing.assert_allclose(h[0], h_full[n_cached:], rtol=1e-11, atol=1e-12)
        np.testing.assert_allclose(k, k_full[:, n_cached:], rtol=1e-11, atol=1e-12)
        np.testing.assert_allclose(v, v_full[:, n_cached:], rtol=1e-11, atol=1e-12)
    # four appends of one token each
    _, kc, vc = prefill(orc, p, x[:5])
    kc, vc = list(kc), list(vc)
    for i in range(5, 9):
        h, k, v = append(orc, p, kc, vc, np.array([0, i]), x[None, i:i + 1])
        kc = [np.concatenate([kc[l], k[l]], 0) for l in range(len(kc))]
        vc = [np.concatenate([vc[l], v[l]], 0) for l in range(len(vc))]
    h_full, k_full, v_full = prefill(orc, p, x[:9])
    np.testing.assert_allclose(h[0, 0], h_full[8], rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(np.stack(kc), k_full, rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(np.stack(vc), v_full, rtol=1e-11, atol=1e-12)


def pin_append_causal(orc):
    """A new token never sees later new tokens: changing the last one leaves the others'
    hidden states and rows unchanged; changing the first one changes every token."""
    p = tiny_params(12)
    r = np.random.default_rng(13)
    kc = [r.normal(size=(5, 2, 8)) for _ in range(2)]
    vc = [r.normal(size=(5, 2, 8)) for _ in range(2)]
    x = tiny_tokens(4, 14)
    h, k, v = append(orc, p, kc, vc, np.array([0, 5]), x[None])
    x2 = x.copy()
    x2[3] += 1.0
    h2, k2, v2 = append(orc, p, kc, vc, np.array([0, 5]), x2[None])
    np.testing.assert_array_equal(h2[0, :3], h[0, :3])
    np.testing.assert_array_equal(k2[:, :3], k[:, :3])
    assert np.max(np.abs(h2[0, 3] - h[0, 3])) > 1e-6
    x3 = x.copy()
    x3[0] += 1.0
    h3, _, _ = append(orc, p, kc, vc, np.array([0, 5]), x3[None])
    assert np.min(np.max(np.abs(h3[0] - h[0]), axis=-1)) > 1e-9


def pin_append_vehicles_and_readonly(orc):
    """Vehicles with ragged caches (one empty) in one call equal separate calls; the
    caches are not written; another vehicle's cache rows do not matter; a vehicle's own
    cache rows do."""
    p = tiny_params(15)
    r = np.random.default_rng(16)
    lengths = [3, 0, 7]
    off = np.concatenate([[0], np.cumsum(lengths)])
    kc = [r.normal(size=(off[-1], 2, 8)) for _ in range(2)]
    vc = [r.normal(size=(off[-1], 2, 8)) for _ in range(2)]
    before = [a.copy() for a in kc + vc]
    x = r.normal(size=(3, 4, TINY["d_model"]))
    h, k, v = append(orc, p, kc, vc, off, x)
    for a, b in zip(kc + vc, before):
        np.testing.assert_array_equal(a, b)
    for b in range(3):
        lo, hi = off[b], off[b + 1]
        hb, kb, vb = append(orc, p, [a[lo:hi] for a in kc], [a[lo:hi] for a in vc], np.array([0, hi - lo]),
                            x[b:b + 1])
        np.testing.assert_allclose(h[b], hb[0], rtol=1e-13, atol=1e-14)
        np.testing.assert_allclose(k[:, 4 * b:4 * b + 4], kb, rtol=1e-13, atol=1e-14)
        np.testing.assert_allclose(v[:, 4 * b:4 * b + 4], vb, rtol=1e-13, atol=1e-14)
    kc2 = [a.copy() for a in kc]
    vc2 = [a.copy() for a in vc]
    for a in kc2 + vc2:
        a[off[2]:off[3]] *= -1.3
    h2, _, _ = append(orc, p, kc2, vc2, off, x)
    np.testing.assert_array_equal(h2[:2], h[:2])
    assert np.max(np.abs(h2[2] - h[2])) > 1e-6


PINS = [pin_rope_complex, pin_rope_closed_forms, pin_prefill_library, pin_append_library,
        pin_incremental_equals_monolithic, pin_append_causal, pin_append_vehicles_and_readonly]


@pytest.mark.parametrize("pin", PINS, ids=lambda f: f.__name__)
def test_pin(pin):
    pin(append_oracle)


# ---------------------------------------------------------------- planted mistakes
MUTATIONS = {
    "rope_sign": ("a * sin + b * cos", "-a * sin + b * cos"),
    "rope_interleaved_pairs": ("a = x[..., :half]\n    b = x[..., half:]", "a = x[..., 0::2]\n    b = x[..., 1::2]"),
    "rope_frequency_exponent": ("base ** (-2.0 * np.arange(half", "base ** (-1.0 * np.arange(half"),
    "append_positions_from_zero": ("pos = n_cached + np.arange(n_app)", "pos = np.arange(n_app)"),
    "append_mask_strict": ("<= (n_cached + np.arange(n_app))", "< (n_cached + np.arange(n_app))"),
    "append_mask_dropped": ("s = np.where(visible, s, -np.inf)", "s = s"),
    "append_cache_keys_dropped": ("k_cache[layer][lo:hi]", "k_cache[layer][lo:lo]"),
    "append_keys_not_rotated": ('k = rope((n @ _layer(params, layer, "wk").T).reshape(n_app, n_heads, head_dim), pos, base)',
                                'k = (n @ _layer(params, layer, "wk").T).reshape(n_app, n_heads, head_dim)'),
    "prefill_mask_transposed": ("np.tril(", "np.triu("),
    "score_scale_dropped": (" / np.sqrt(head_dim)", ""),
    "prefill_values_rotated": ('v = (n @ _layer(params, layer, "wv").T).reshape(s_len, n_heads, head_dim)',
                               'v = rope((n @ _layer(params, layer, "wv").T).reshape(s_len, n_heads, head_dim), pos, base)'),
    "append_attn_residual_dropped": ("x = x + a.reshape(n_app, hd)", "x = a.reshape(n_app, hd)"),
    "append_mlp_gate_up_swapped": ('(silu(n @ _layer(params, layer, "w_gate").T) * (n @ _layer(params, layer, "w_up").T)) \\\n                @',
                                   '(silu(n @ _layer(params, layer, "w_up").T) * (n @ _layer(params, layer, "w_gate").T)) \\\n                @'),
}


def _mutant(name):
    src_path = append_oracle.__file__
    with open(src_path) as fh:
        src = fh.read()
    old, new = MUTATIONS[name]
    assert src.count(old) >= 1, f"mutation {name!r} no longer matches the oracle source"
    mod = types.ModuleType(f"oracle.append_mutant_{name}")
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
