"""The seeded input recipe and the bench's roofline arithmetic, checked on the CPU.

The synthetic inputs must have the shapes and distributions the workloads state:
  projection weights N(0, 1/fan_in), norm gains 1 + 0.1 N(0, 1), embeddings
  N(0, 0.02^2), frames N(0, 1), cache K = N(0, 1) * s with s ~ LogNormal(0, 0.5)
  per (layer, head, dim), cache V N(0, 1), bf16 rounding for "bf16" workloads,
  ragged cache lengths uniform in the stated ranges.
The roofline figures of bench.py must equal the byte and FLOP counts worked out by
hand from the shapes.
"""
from __future__ import annotations

import math
import os
import sys

import numpy as np
import torch

from paper_2607_15621_gb300 import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)
import bench  # noqa: E402

SMALL = synth.Dims(n_layers=2, d_model=256, n_heads=4, d_ff=384)


def test_expert_weight_distributions_and_bf16_rounding():
    w = synth.make_weights(SMALL, 0, "bf16")
    d, hd, f = SMALL.d_model, SMALL.hd, SMALL.d_ff
    assert w["wq"].shape == (2, hd, d) and w["wo"].shape == (2, d, hd) and w["w_down"].shape == (2, d, f)
    for name, fan_in in (("wq", d), ("wk", d), ("wv", d), ("wo", hd), ("w_gate", d), ("w_up", d), ("w_down", f)):
        assert abs(w[name].std() * math.sqrt(fan_in) - 1.0) < 0.02, name
        assert abs(w[name].mean()) * math.sqrt(fan_in) < 0.02, name
    for name in ("attn_norm", "mlp_norm", "final_norm"):
        assert abs(w[name].mean() - 1.0) < 0.02 and abs(w[name].std() - 0.1) < 0.02, name
    assert abs(w["act_emb"].std() - 0.02) < 0.004 and abs(w["pos_emb"].std() - 0.02) < 0.004
    for v in w.values():  # every value is a bf16 number
        t = torch.as_tensor(v)
        assert torch.equal(t, t.to(torch.bfloat16).to(torch.float32))
    w2 = synth.make_weights(SMALL, 0, "bf16")
    assert all(np.array_equal(w[k], w2[k]) for k in w)  # seeded


def test_cache_distributions():
    lengths = [3000, 1000]
    k, v, off = synth.make_cache(SMALL, lengths, 0, "fp32")
    assert list(off) == [0, 3000, 4000]
    assert k[0].shape == (4000, SMALL.n_heads, SMALL.head_dim) and k[0].dtype == torch.float32
    for layer in range(SMALL.n_layers):
        scale = k[layer].std(dim=0)                       # per (head, dim): the LogNormal factor
        ls = torch.log(scale)
        assert abs(ls.mean().item()) < 0.06 and abs(ls.std().item() - 0.5) < 0.05
        z = k[layer] / scale
        assert abs(z.std().item() - 1.0) < 0.01
        assert abs(v[layer].std().item() - 1.0) < 0.01 and abs(v[layer].mean().item()) < 0.01
    kb, vb, _ = synth.make_cache(SMALL, [10], 0, "bf16")
    assert kb[0].dtype == torch.bfloat16 and vb[0].dtype == torch.bfloat16


def test_frames_and_lengths():
    fr = synth.make_frames(SMALL, 64, 0, "fp32")
    assert fr.shape == (64, SMALL.n_frame, SMALL.d_model)
    assert abs(fr.std().item() - 1.0) < 0.01 and abs(fr.mean().item()) < 0.01
    for name, lo, hi, b in (("bf16_b16_ragged", 96, 480, 16), ("bf16_b128_ragged", 64, 2048, 128)):
        L = synth.cache_lengths(name, 0)
        assert len(L) == b and L.min() >= lo and L.max() <= hi
        assert np.array_equal(L, synth.cache_lengths(name, 0))
    assert list(synth.cache_lengths("bf16_b1_l224", 0)) == [224]
    # the large fleet draw that the measurements quote
    assert int(synth.cache_lengths("bf16_b128_ragged", 0).sum()) == 129767


def test_backbone_weights_and_append_tokens():
    dims = synth.BackboneDims(n_layers=1, d_model=256, n_heads=2, d_ff=384)
    w = synth.make_backbone_weights(dims, 0, "bf16")
    assert w["wq"].shape == (1, dims.hd, dims.d_model) and w["w_down"].shape == (1, dims.d_model, dims.d_ff)
    assert abs(w["wq"].std() * math.sqrt(dims.d_model) - 1.0) < 0.03
    assert abs(w["w_down"].std() * math.sqrt(dims.d_ff) - 1.0) < 0.03
    x = synth.make_append_tokens(dims, 8, 0)
    assert x.shape == (8, dims.n_new, dims.d_model) and x.dtype == torch.bfloat16
    assert abs(x.float().std().item() - 1.0) < 0.03


def test_tick_roofline_arithmetic():
    """Bytes per tick = expert weights once + every cached row once per layer; FLOPs =
    projections (2 per weight and token) + Eq. 1 (4 T D per key, head and layer)."""
    dims = synth.EXPERT
    w_bytes = 675_282_944  # the fp16 weight arena of the 32-layer expert: 10,551,296 x 2 B x 32 layers
    by, kv = bench.algorithmic_bytes(dims, [224], "bf16", w_bytes)
    assert kv == 224 * 32 * 2 * 4096 * 2
    assert by == w_bytes + kv == 792_723_456  # the bench line's bytes per tick at B = 1, L = 224
    assert w_bytes == 10_551_296 * 2 * 32
    per_layer_w = 3 * 4096 * 512 + 512 * 4096 + 2 * 1408 * 512 + 512 * 1408
    assert per_layer_w == 10_551_296
    flops = bench.tick_flops(dims, [224])
    assert flops == 2 * 42 * per_layer_w * 32 + 4 * 42 * 128 * 32 * (224 + 42) * 32
    # B = 1, L = 224: 28.36 GFLOP of projections (the figure the workload analysis quotes)
    assert abs(2 * 42 * per_layer_w * 32 / 1e9 - 28.36) < 0.01
    by32, kv32 = bench.algorithmic_bytes(dims, [96], "fp32", w_bytes)
    assert kv32 == 96 * 32 * 2 * 4096 * 4


def test_clip_prefixes_follow_the_visibility_rule():
    """The clip workload's per-block prefixes are the oracle's visible prefixes (Sec. 3.2)."""
    from oracle import staleness_oracle
    c = synth.CLIP_WORKLOADS["clip_j40_delta1"]
    got = synth.clip_prefixes("clip_j40_delta1")
    want = [staleness_oracle.visible_prefix(j, c["delta"], c["text"], c["tokens_per_frame"]) for j in range(c["frames"])]
    assert list(got) == want
    assert got.max() <= c["text"] + c["tokens_per_frame"] * c["frames"]


def test_paper_layout_recipe():
    """Ten-token layout inputs: the layer stack of make_weights plus the state MLP, queries,
    positions and the two-layer head with the stated scales; ego state and visual tokens
    N(0, 1)."""
    import math
    from paper_2607_15621_gb300 import synth
    dims = synth.Dims(n_layers=2, n_action=5, n_frame=5)
    w = synth.make_paper_weights(dims, 0, "fp32")
    base = synth.make_weights(dims, 0, "fp32")
    assert np.array_equal(w["wq"], base["wq"]) and np.array_equal(w["final_norm"], base["final_norm"])
    d = dims.d_model
    shapes = {"state_w1": (d, 16), "state_w2": (d, d), "query_emb": (5, d), "pos_emb": (10, d), "head_w1": (d, d),
              "head_w2": (2, d), "head_b2": (2,)}
    for k, shp in shapes.items():
        assert w[k].shape == shp, k
    assert abs(w["state_w1"].std() - 1 / 4) < 0.02
    assert abs(w["state_w2"].std() - 1 / math.sqrt(d)) < 0.003
    assert abs(w["head_w1"].std() - 1 / math.sqrt(d)) < 0.003
    assert abs(w["query_emb"].std() - 0.02) < 0.002 and abs(w["pos_emb"].std() - 0.02) < 0.002
    assert "act_emb" not in w and "head_w" not in w
    visual, state = synth.make_paper_inputs(dims, 3, 0, "bf16")
    assert visual.shape == (3, 4, d) and visual.dtype == torch.bfloat16 and state.shape == (3, 16)
    assert abs(float(visual.float().std()) - 1.0) < 0.05
    v2, s2 = synth.make_paper_inputs(dims, 3, 0, "bf16")
    assert torch.equal(visual, v2) and torch.equal(state, s2)
