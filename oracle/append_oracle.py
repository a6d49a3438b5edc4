"""Plain fp64 CPU oracle of the backbone's incremental cache append.

TEST INFRASTRUCTURE, like ``fsx_oracle``: only ``tests/``,
``__graft_entry__.smoke()`` and ``bench.py``'s CPU legs may import it; it takes
and returns plain numpy arrays and imports nothing from the product path.

What it computes (Sec. 1 and Sec. 3.3, "Asynchronous Deployment"): every K = 4
ticks the slow system appends the current frame's four tokens to the frozen
backbone's per-layer key-value cache with an incremental forward pass whose
cost does not depend on the history length. Rotary phases make the append
exact: the rows it appends, and the hidden states it produces, equal those of a
monolithic forward over the whole sequence (the paper's golden equivalence
test compares the two). Two plain definitions are written here so that this
equivalence can be checked between them:

  backbone_prefill  the monolithic causal forward over one whole sequence;
  backbone_append   the incremental forward of A new tokens per vehicle over
                    an existing cache (the vehicle's rows [offsets[b],
                    offsets[b+1]) of every layer), returning the K/V rows to
                    append at positions L_b .. L_b + A - 1.

Layer (LLaMA-style decoder, in the paper's backbone order), for token rows X:
  N = RMSNorm(X, g1);  Q = N W_q^T,  K = N W_k^T,  V = N W_v^T      (H heads of D)
  Q, K <- RoPE(Q, pos), RoPE(K, pos)
  A = softmax(Q [K_cache ; K]^T / sqrt(D) + causal mask) [V_cache ; V]
  X = X + A W_o^T;  N = RMSNorm(X, g2);  X = X + (silu(N W_g^T) * (N W_u^T)) W_d^T

Readings where the paper is silent (the backbone is LMDrive's frozen LLaMA-7B):
  * shape: 32 layers, d = 4096, 32 heads of 128, SwiGLU hidden 11008, no
    biases, pre-norm RMSNorm with eps = 1e-6 (the LLaMA convention);
  * RoPE with base 10000 on queries and keys, pairing dims j and j + D/2 of a
    head (the rotate-half convention), angle pos * base^(-2j/D); the cache
    stores keys after the rotation, values as computed;
  * a vehicle's cached token i sits at position i (the cache holds the whole
    history from position 0), so the appended tokens take positions
    L_b .. L_b + A - 1;
  * causal attention: appended token i sees every cached row of its vehicle
    and appended tokens 0 .. i of the same vehicle; vehicles never see each
    other;
  * the returned hidden states are the residual stream after the last layer
    (no final norm); the paper's episode-boundary head is not specified.

Parity status: every function is pinned in tests/test_append_oracle_pins.py
(torch SDPA with an explicit mask, RoPE as complex multiplication, closed
forms, the monolithic/incremental equivalence the paper states, causality and
independence invariants).
"""
from __future__ import annotations

import numpy as np

from .fsx_oracle import RMS_EPS, rms_norm, silu

ROPE_BASE = 10000.0


def rope(x: np.ndarray, positions, base: float = ROPE_BASE) -> np.ndarray:
    """Rotary position embedding of x [S, H, D] (D even) at integer positions [S].

    Dims j and j + D/2 of every head form a pair rotated by the angle
    positions[s] * base^(-2j/D), j = 0 .. D/2 - 1."""
    x = np.asarray(x, dtype=np.float64)
    pos = np.asarray(positions, dtype=np.float64)
    d = x.shape[-1]
    half = d // 2
    inv_freq = base ** (-2.0 * np.arange(half, dtype=np.float64) / d)   # [D/2]
    ang = pos[:, None] * inv_freq[None, :]                              # [S, D/2]
    cos = np.cos(ang)[:, None, :]
    sin = np.sin(ang)[:, None, :]
    a = x[..., :half]
    b = x[..., half:]
    return np.concatenate([a * cos - b * sin, a * sin + b * cos], axis=-1)


def _layer(params: dict, layer: int, name: str) -> np.ndarray:
    return np.asarray(params[name][layer], dtype=np.float64)


def _softmax_rows(s: np.ndarray) -> np.ndarray:
    m = np.max(s, axis=-1, keepdims=True)
    e = np.exp(s - m)
    return e / np.sum(e, axis=-1, keepdims=True)


def backbone_prefill(params: dict, x: np.ndarray, n_heads: int, head_dim: int,
                     base: float = ROPE_BASE, eps: float = RMS_EPS):
    """Monolithic causal forward over one sequence of S token embeddings x [S, d].

    params: stacked over layers, matrices [out_features, in_features]:
      attn_norm [NL, d], wq/wk/wv [NL, H*D, d], wo [NL, d, H*D],
      mlp_norm [NL, d], w_gate/w_up [NL, F, d], w_down [NL, d, F].
    Returns (h [S, d], k [NL, S, H, D], v [NL, S, H, D]): the residual stream
    after the last layer and every layer's cache rows (keys after RoPE)."""
    x = np.array(x, dtype=np.float64)
    s_len = x.shape[0]
    n_layers = len(params["wq"])
    hd = n_heads * head_dim
    pos = np.arange(s_len)
    k_all = np.zeros((n_layers, s_len, n_heads, head_dim))
    v_all = np.zeros((n_layers, s_len, n_heads, head_dim))
    if s_len == 0:  # an empty sequence leaves an empty cache
        return x, k_all, v_all
    for layer in range(n_layers):
        n = rms_norm(x, _layer(params, layer, "attn_norm"), eps)
        q = rope((n @ _layer(params, layer, "wq").T).reshape(s_len, n_heads, head_dim), pos, base)
        k = rope((n @ _layer(params, layer, "wk").T).reshape(s_len, n_heads, head_dim), pos, base)
        v = (n @ _layer(params, layer, "wv").T).reshape(s_len, n_heads, head_dim)
        k_all[layer] = k
        v_all[layer] = v
        a = np.zeros((s_len, n_heads, head_dim))
        for h in range(n_heads):
            s = q[:, h, :] @ k[:, h, :].T / np.sqrt(head_dim)            # [S, S]
            s = np.where(np.tril(np.ones((s_len, s_len), dtype=bool)), s, -np.inf)
            a[:, h, :] = _softmax_rows(s) @ v[:, h, :]
        x = x + a.reshape(s_len, hd) @ _layer(params, layer, "wo").T
        n = rms_norm(x, _layer(params, layer, "mlp_norm"), eps)
        x = x + (silu(n @ _layer(params, layer, "w_gate").T) * (n @ _layer(params, layer, "w_up").T)) \
            @ _layer(params, layer, "w_down").T
    return x, k_all, v_all


def backbone_append(params: dict, k_cache, v_cache, offsets, x_new: np.ndarray, n_heads: int, head_dim: int,
                    base: float = ROPE_BASE, eps: float = RMS_EPS):
    """Incremental forward of A new tokens per vehicle over the existing cache.

    k_cache, v_cache: NL arrays [total_tokens, H, D]; vehicle b owns rows
      offsets[b] .. offsets[b+1]-1 (its tokens 0 .. L_b-1). They are only read.
    offsets: [B+1] non-decreasing integers.
    x_new: [B, A, d] embeddings of the tokens to append.
    Returns (h [B, A, d], k_new [NL, B*A, H, D], v_new [NL, B*A, H, D]): the
    residual stream after the last layer and, per layer, the rows to append
    (vehicle-major, keys after RoPE at positions L_b .. L_b + A - 1)."""
    x_new = np.array(x_new, dtype=np.float64)
    offsets = np.asarray(offsets, dtype=np.int64)
    n_batch, n_app, _ = x_new.shape
    n_layers = len(params["wq"])
    hd = n_heads * head_dim
    k_out = np.zeros((n_layers, n_batch * n_app, n_heads, head_dim))
    v_out = np.zeros((n_layers, n_batch * n_app, n_heads, head_dim))
    h_out = np.zeros_like(x_new)
    for b in range(n_batch):
        lo, hi = int(offsets[b]), int(offsets[b + 1])
        n_cached = hi - lo
        pos = n_cached + np.arange(n_app)                 # positions of the new tokens
        x = x_new[b].copy()
        for layer in range(n_layers):
            n = rms_norm(x, _layer(params, layer, "attn_norm"), eps)
            q = rope((n @ _layer(params, layer, "wq").T).reshape(n_app, n_heads, head_dim), pos, base)
            k = rope((n @ _layer(params, layer, "wk").T).reshape(n_app, n_heads, head_dim), pos, base)
            v = (n @ _layer(params, layer, "wv").T).reshape(n_app, n_heads, head_dim)
            k_out[layer, b * n_app:(b + 1) * n_app] = k
            v_out[layer, b * n_app:(b + 1) * n_app] = v
            k_keys = np.concatenate([np.asarray(k_cache[layer][lo:hi], np.float64), k], axis=0)
            v_keys = np.concatenate([np.asarray(v_cache[layer][lo:hi], np.float64), v], axis=0)
            # new token i sees cached rows 0 .. L_b-1 and new tokens 0 .. i
            visible = np.arange(n_cached + n_app)[None, :] <= (n_cached + np.arange(n_app))[:, None]
            a = np.zeros((n_app, n_heads, head_dim))
            for h in range(n_heads):
                s = q[:, h, :] @ k_keys[:, h, :].T / np.sqrt(head_dim)     # [A, L_b + A]
                s = np.where(visible, s, -np.inf)
                a[:, h, :] = _softmax_rows(s) @ v_keys[:, h, :]
            x = x + a.reshape(n_app, hd) @ _layer(params, layer, "wo").T
            n = rms_norm(x, _layer(params, layer, "mlp_norm"), eps)
            x = x + (silu(n @ _layer(params, layer, "w_gate").T) * (n @ _layer(params, layer, "w_up").T)) \
                @ _layer(params, layer, "w_down").T
        h_out[b] = x
    return h_out, k_out, v_out
