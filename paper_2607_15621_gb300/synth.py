"""Seeded synthetic inputs for the action-expert tick.

This module only draws random numbers with fixed shapes and distributions; it
holds none of the expert's arithmetic. Both the CUDA path's tests/bench and the
oracle's tests consume what it produces, so it imports neither of them.

Distributions (one recipe for every workload):
  expert weights  W ~ N(0, 1/fan_in) for every projection, head W_h ~ N(0, 1/d),
                  head bias ~ N(0, 0.1^2)
  norm gains      gamma ~ 1 + 0.1 N(0, 1)
  embeddings      action / positional ~ N(0, 0.02^2)
  frame tokens    ~ N(0, 1)
  cache keys      K ~ N(0, 1) * s[l, h, d], s ~ LogNormal(0, 0.5) drawn once per layer
  cache values    V ~ N(0, 1)
For "bf16" workloads every weight, cache row and frame token is rounded to
bfloat16 (round-to-nearest-even) as part of the input, so the oracle and the
CUDA path read the same values. For "fp32" workloads the inputs stay fp32.
"""
from __future__ import annotations

import math
from dataclasses import dataclass

import numpy as np
import torch


@dataclass(frozen=True)
class Dims:
    n_layers: int = 32
    d_model: int = 512
    n_heads: int = 32
    head_dim: int = 128
    d_ff: int = 1408
    n_action: int = 10
    n_frame: int = 32
    n_waypoints: int = 5

    @property
    def n_tok(self) -> int:
        return self.n_action + self.n_frame

    @property
    def hd(self) -> int:
        return self.n_heads * self.head_dim

    def n_params(self) -> int:
        d, hd, f, nl = self.d_model, self.hd, self.d_ff, self.n_layers
        per_layer = 3 * hd * d + d * hd + 2 * f * d + d * f + 2 * d
        return nl * per_layer + self.n_action * d + self.n_tok * d + d + 2 * d + 2


EXPERT = Dims()


@dataclass(frozen=True)
class BackboneDims:
    """Shape of the frozen backbone whose cache the slow system appends to
    (a LLaMA-7B-shaped causal decoder) and of one append call."""
    n_layers: int = 32
    d_model: int = 4096
    n_heads: int = 32
    head_dim: int = 128
    d_ff: int = 11008
    n_new: int = 4
    rope_base: float = 10000.0

    @property
    def hd(self) -> int:
        return self.n_heads * self.head_dim


BACKBONE = BackboneDims()

# Staleness-masked clip workloads (Sec. 3.2): one clip cache of `text` instruction rows
# plus `frames` x 4 frame rows; frame j's expert block reads the prefix ending `delta`
# frames earlier, and all blocks run as one batched tick over explicit row ranges.
CLIP_WORKLOADS = {
    "clip_j40_delta1": dict(text=64, frames=40, delta=1, tokens_per_frame=4),
}


def clip_prefixes(workload: str) -> np.ndarray:
    """Cache rows visible to each frame block of a clip workload (text, plus frames 0 .. j - delta)."""
    c = CLIP_WORKLOADS[workload]
    j = np.arange(c["frames"])
    return np.where(j < c["delta"], c["text"], c["text"] + c["tokens_per_frame"] * (j - c["delta"] + 1)).astype(np.int64)


# Cache-append workloads: one call appends n_new tokens for each of `batch`
# vehicles, each with `length` cached tokens (64 instruction + 40 frames x 4).
APPEND_WORKLOADS = {
    "append_b1_l224": dict(batch=1, length=224),
}

# The asynchronous fast-slow schedule (Sec. 3.3): one vehicle with `length` cached tokens,
# a tick every `cadence_ms` and an append of 4 tokens before every `k`-th tick.
FASTSLOW_WORKLOADS = {
    "fastslow_b1_l224": dict(length=224, k=4, cadence_ms=12.5),
}

# The paper's ten-token layout (Sec. 3.1): `batch` vehicles, each with `length` cached tokens.
PAPER_WORKLOADS = {
    "paper_b1_l224": dict(batch=1, length=224),
}

# Workloads: name -> (batch, length spec, dtype). Length spec is either a fixed
# per-vehicle cache length or a (lo, hi) inclusive uniform range.
WORKLOADS = {
    "fp32_b1_l96": dict(batch=1, length=96, dtype="fp32"),
    "bf16_b1_l224": dict(batch=1, length=224, dtype="bf16"),
    "bf16_b1_l512": dict(batch=1, length=512, dtype="bf16"),
    "bf16_b1_l1024": dict(batch=1, length=1024, dtype="bf16"),
    "bf16_b1_l2048": dict(batch=1, length=2048, dtype="bf16"),
    "bf16_b1_l4096": dict(batch=1, length=4096, dtype="bf16"),
    "bf16_b16_ragged": dict(batch=16, length=(96, 480), dtype="bf16"),
    "bf16_b128_ragged": dict(batch=128, length=(64, 2048), dtype="bf16"),
}

_STREAM_WEIGHTS = 0x5EED0001
_STREAM_CACHE = 0x5EED0002
_STREAM_FRAMES = 0x5EED0003
_STREAM_LENGTHS = 0x5EED0004
_STREAM_BACKBONE = 0x5EED0005
_STREAM_APPEND_TOKENS = 0x5EED0006
_STREAM_PAPER_WEIGHTS = 0x5EED0007
_STREAM_PAPER_INPUTS = 0x5EED0008


def _gen(seed: int, stream: int, device="cpu") -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed((int(seed) * 1_000_003 + stream) & 0x7FFF_FFFF_FFFF_FFFF)
    return g


def _round(t: torch.Tensor, dtype: str) -> torch.Tensor:
    if dtype == "bf16":
        return t.to(torch.bfloat16).to(torch.float32)
    if dtype == "fp32":
        return t
    raise ValueError(f"unknown dtype {dtype!r}")


def make_weights(dims: Dims = EXPERT, seed: int = 0, dtype: str = "fp32") -> dict:
    """Expert weights as C-contiguous float32 numpy arrays, stacked over layers.

    Matrices are [out_features, in_features]."""
    g = _gen(seed, _STREAM_WEIGHTS)
    nl, d, hd, f = dims.n_layers, dims.d_model, dims.hd, dims.d_ff

    def normal(shape, std):
        return torch.randn(*shape, generator=g, dtype=torch.float32) * std

    w = {
        "act_emb": normal((dims.n_action, d), 0.02),
        "pos_emb": normal((dims.n_tok, d), 0.02),
        "attn_norm": 1.0 + normal((nl, d), 0.1),
        "wq": normal((nl, hd, d), 1.0 / math.sqrt(d)),
        "wk": normal((nl, hd, d), 1.0 / math.sqrt(d)),
        "wv": normal((nl, hd, d), 1.0 / math.sqrt(d)),
        "wo": normal((nl, d, hd), 1.0 / math.sqrt(hd)),
        "mlp_norm": 1.0 + normal((nl, d), 0.1),
        "w_gate": normal((nl, f, d), 1.0 / math.sqrt(d)),
        "w_up": normal((nl, f, d), 1.0 / math.sqrt(d)),
        "w_down": normal((nl, d, f), 1.0 / math.sqrt(f)),
        "final_norm": 1.0 + normal((d,), 0.1),
        "head_w": normal((2, d), 1.0 / math.sqrt(d)),
        "head_b": normal((2,), 0.1),
    }
    return {k: np.ascontiguousarray(_round(v, dtype).numpy()) for k, v in w.items()}


def cache_lengths(workload: str, seed: int = 0) -> np.ndarray:
    spec = WORKLOADS[workload]
    batch, length = spec["batch"], spec["length"]
    if isinstance(length, int):
        return np.full(batch, length, dtype=np.int64)
    lo, hi = length
    g = _gen(seed, _STREAM_LENGTHS)
    return torch.randint(lo, hi + 1, (batch,), generator=g).numpy().astype(np.int64)


def offsets_from_lengths(lengths) -> np.ndarray:
    lengths = np.asarray(lengths, dtype=np.int64)
    return np.concatenate([[0], np.cumsum(lengths)]).astype(np.int64)


def make_cache(dims: Dims, lengths, seed: int = 0, dtype: str = "bf16", device="cpu"):
    """Per-layer backbone KV cache, token-major [sum(L_b), H, D] per layer.

    Returns (k_layers, v_layers, offsets) with torch tensors on ``device``
    (bfloat16 for "bf16", float32 for "fp32") and int64 numpy offsets."""
    offsets = offsets_from_lengths(lengths)
    total = int(offsets[-1])
    dev = torch.device(device)
    g = _gen(seed, _STREAM_CACHE, device=dev.type if dev.type == "cpu" else dev)
    store = torch.bfloat16 if dtype == "bf16" else torch.float32
    k_layers, v_layers = [], []
    for _ in range(dims.n_layers):
        scale = torch.exp(0.5 * torch.randn(dims.n_heads, dims.head_dim, generator=g, device=dev))
        k = torch.randn(total, dims.n_heads, dims.head_dim, generator=g, device=dev) * scale
        v = torch.randn(total, dims.n_heads, dims.head_dim, generator=g, device=dev)
        k_layers.append(k.to(store).contiguous())
        v_layers.append(v.to(store).contiguous())
    return k_layers, v_layers, offsets


def make_frames(dims: Dims, batch: int, seed: int = 0, dtype: str = "bf16", device="cpu"):
    """Frame tokens [B, n_frame, d] (bfloat16 for "bf16", float32 for "fp32")."""
    dev = torch.device(device)
    g = _gen(seed, _STREAM_FRAMES, device=dev.type if dev.type == "cpu" else dev)
    f = torch.randn(batch, dims.n_frame, dims.d_model, generator=g, device=dev)
    return f.to(torch.bfloat16 if dtype == "bf16" else torch.float32).contiguous()


def as_f64(t: torch.Tensor) -> np.ndarray:
    """Exact fp64 copy of a (possibly bf16 / device) tensor for the oracle."""
    return t.detach().to("cpu", torch.float64).numpy()


def make_backbone_weights(dims: BackboneDims = BACKBONE, seed: int = 0, dtype: str = "bf16") -> dict:
    """Backbone weights as C-contiguous float32 numpy arrays, stacked over layers,
    [out_features, in_features]: W ~ N(0, 1/fan_in), norm gains ~ 1 + 0.1 N(0, 1)."""
    g = _gen(seed, _STREAM_BACKBONE)
    nl, d, hd, f = dims.n_layers, dims.d_model, dims.hd, dims.d_ff

    def normal(shape, std):
        return torch.randn(*shape, generator=g, dtype=torch.float32) * std

    w = {
        "attn_norm": 1.0 + normal((nl, d), 0.1),
        "wq": normal((nl, hd, d), 1.0 / math.sqrt(d)),
        "wk": normal((nl, hd, d), 1.0 / math.sqrt(d)),
        "wv": normal((nl, hd, d), 1.0 / math.sqrt(d)),
        "wo": normal((nl, d, hd), 1.0 / math.sqrt(hd)),
        "mlp_norm": 1.0 + normal((nl, d), 0.1),
        "w_gate": normal((nl, f, d), 1.0 / math.sqrt(d)),
        "w_up": normal((nl, f, d), 1.0 / math.sqrt(d)),
        "w_down": normal((nl, d, f), 1.0 / math.sqrt(f)),
    }
    return {k: np.ascontiguousarray(_round(v, dtype).numpy()) for k, v in w.items()}


def make_append_tokens(dims: BackboneDims, batch: int, seed: int = 0, device="cpu"):
    """Embeddings of the tokens one append call adds, bf16 [B, n_new, d] ~ N(0, 1)."""
    dev = torch.device(device)
    g = _gen(seed, _STREAM_APPEND_TOKENS, device=dev.type if dev.type == "cpu" else dev)
    x = torch.randn(batch, dims.n_new, dims.d_model, generator=g, device=dev)
    return x.to(torch.bfloat16).contiguous()


PAPER_STATE_DIM = 16
PAPER_VISUAL = 4
PAPER_QUERIES = 5


def make_paper_weights(dims: Dims = EXPERT, seed: int = 0, dtype: str = "fp32") -> dict:
    """Weights of the paper's ten-token layout: the layer stack of make_weights (same seed)
    plus the state MLP (W_s1 ~ N(0, 1/16), W_s2 ~ N(0, 1/d), biases ~ N(0, 0.1^2)), the
    five waypoint queries and the [10, d] position table (~ N(0, 0.02^2)), and the
    two-layer head (W_h1 ~ N(0, 1/d), W_h2 ~ N(0, 1/d), biases ~ N(0, 0.1^2))."""
    base = make_weights(dims, seed, dtype)
    g = _gen(seed, _STREAM_PAPER_WEIGHTS)
    d = dims.d_model

    def normal(shape, std):
        return torch.randn(*shape, generator=g, dtype=torch.float32) * std

    extra = {
        "state_w1": normal((d, PAPER_STATE_DIM), 1.0 / math.sqrt(PAPER_STATE_DIM)),
        "state_b1": normal((d,), 0.1),
        "state_w2": normal((d, d), 1.0 / math.sqrt(d)),
        "state_b2": normal((d,), 0.1),
        "query_emb": normal((PAPER_QUERIES, d), 0.02),
        "pos_emb": normal((1 + PAPER_VISUAL + PAPER_QUERIES, d), 0.02),
        "head_w1": normal((d, d), 1.0 / math.sqrt(d)),
        "head_b1": normal((d,), 0.1),
        "head_w2": normal((2, d), 1.0 / math.sqrt(d)),
        "head_b2": normal((2,), 0.1),
    }
    w = {k: v for k, v in base.items() if k not in ("act_emb", "pos_emb", "head_w", "head_b")}
    w.update({k: np.ascontiguousarray(_round(v, dtype).numpy()) for k, v in extra.items()})
    return w


def make_paper_inputs(dims: Dims, batch: int, seed: int = 0, dtype: str = "bf16", device="cpu"):
    """Visual tokens [B, 4, d] (bfloat16 for "bf16", float32 for "fp32") ~ N(0, 1) and the
    fp32 ego state [B, 16] ~ N(0, 1) of the ten-token layout."""
    dev = torch.device(device)
    g = _gen(seed, _STREAM_PAPER_INPUTS, device=dev.type if dev.type == "cpu" else dev)
    visual = torch.randn(batch, PAPER_VISUAL, dims.d_model, generator=g, device=dev)
    state = torch.randn(batch, PAPER_STATE_DIM, generator=g, device=dev)
    return visual.to(torch.bfloat16 if dtype == "bf16" else torch.float32).contiguous(), state.contiguous()
