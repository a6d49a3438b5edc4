"""Plain fp64 CPU oracle of the action-expert tick.

TEST INFRASTRUCTURE. Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import this
module. The product path (the ``paper_2607_15621_gb300`` package and its CUDA
library) never imports, links or calls it, and this module imports nothing from
the product path: it takes plain numpy arrays and returns plain numpy arrays.

What it computes (Sec. 3.1 "Action Expert with Per-Layer Cache Attention",
Eq. 1; Sec. 3.3 for the read-only cache): one forward pass of the action
expert for B independent vehicles. Every step is written as its definition, in
the paper's order, in float64, with numpy matmul as the only library primitive:

  X_b      = [E_act ; F_b] + P_pos                                (token assembly)
  for layer l = 0 .. n_layers-1:                (expert layer l reads backbone layer l)
     N          = RMSNorm(X, g1_l)
     Q_ae       = N W_q^l^T,  K_ae = N W_k^l^T,  V_ae = N W_v^l^T  (rectangular projections)
     A          = Attn(Q_ae, [K_vlm^l ; K_ae], [V_vlm^l ; V_ae])   (Eq. 1, per head)
     X          = X + A W_o^l^T                                   (output projection)
     N          = RMSNorm(X, g2_l)
     X          = X + (silu(N W_g^l^T) * (N W_u^l^T)) W_d^l^T       (SwiGLU block)
  waypoint_j = W_h RMSNorm(X_j, g_f) + b_h,  j = 0 .. n_waypoints-1  (waypoint head)

Readings where the paper is silent or where the workload fixes a choice:
  * token layout: ``n_action`` learned action tokens followed by ``n_frame`` frame
    tokens per vehicle (10 + 32 = 42 in the benchmark workloads); the paper's own
    expert uses 10 tokens (1 state + 4 visual + 5 queries, Sec. 3.1). Both are
    just shapes here.
  * pre-norm RMSNorm before attention and before the MLP, a final RMSNorm before
    the head, eps = 1e-6; the paper names no normalisation.
  * attention scale 1/sqrt(head_dim), no bias, no mask, no rotary phase on the
    expert's queries/keys; cached keys are used exactly as stored (Sec. 3.1
    states that backbone keys keep the rotary phases they were cached with).
  * head: one Linear(d -> 2) with bias applied to action tokens 0..n_waypoints-1
    (the paper's "two-layer head" is not specified further).
  * vehicles never attend to each other; vehicle b sees only its own cache
    rows [offsets[b], offsets[b+1]) of every layer.

Parity status: every function here is pinned in tests/test_oracle_pins.py
against library routines (torch scaled_dot_product_attention, rms_norm, silu,
linear), closed forms and invariants; no function is unpinned.
"""
from __future__ import annotations

import numpy as np

RMS_EPS = 1e-6


def rms_norm(x: np.ndarray, gamma: np.ndarray, eps: float = RMS_EPS) -> np.ndarray:
    """RMSNorm over the last axis: x / sqrt(mean(x^2) + eps) * gamma (fp64).

    Applied before attention, before the SwiGLU block and before the head
    (the pre-norm reading of Sec. 3.1's transformer layer)."""
    x = np.asarray(x, dtype=np.float64)
    ms = np.mean(x * x, axis=-1, keepdims=True)
    return x / np.sqrt(ms + eps) * np.asarray(gamma, dtype=np.float64)


def silu(z: np.ndarray) -> np.ndarray:
    """SiLU gate of the SwiGLU feed-forward block (Sec. 3.1): z * sigmoid(z)."""
    z = np.asarray(z, dtype=np.float64)
    return z / (1.0 + np.exp(-z))


def attention_eq1(q_ae, k_vlm, v_vlm, k_ae, v_ae, return_lse: bool = False):
    """Eq. 1 for one vehicle at one layer, every head.

    q_ae  [Tq, H, D]  expert queries
    k_vlm [L,  H, D]  backbone cache keys of this layer (L may be 0)
    v_vlm [L,  H, D]  backbone cache values
    k_ae  [Tk, H, D]  expert keys,  v_ae [Tk, H, D] expert values
    Returns A [Tq, H, D] = softmax(q_ae [K_vlm; K_ae]^T / sqrt(D)) [V_vlm; V_ae]
    per head, and optionally the natural-log log-sum-exp of the scaled scores,
    lse [H, Tq]. The keys are the concatenation (cache first, own tokens
    second); every query sees every key (no mask).
    """
    q = np.asarray(q_ae, dtype=np.float64)
    k_all = np.concatenate([np.asarray(k_vlm, np.float64), np.asarray(k_ae, np.float64)], axis=0)
    v_all = np.concatenate([np.asarray(v_vlm, np.float64), np.asarray(v_ae, np.float64)], axis=0)
    tq, n_heads, d = q.shape
    out = np.empty((tq, n_heads, d), dtype=np.float64)
    lse = np.empty((n_heads, tq), dtype=np.float64)
    scale = 1.0 / np.sqrt(d)
    for h in range(n_heads):
        s = (q[:, h, :] @ k_all[:, h, :].T) * scale          # [Tq, L+Tk]
        m = np.max(s, axis=1, keepdims=True)
        e = np.exp(s - m)
        z = np.sum(e, axis=1, keepdims=True)
        p = e / z                                            # softmax rows
        out[:, h, :] = p @ v_all[:, h, :]
        lse[h, :] = (m + np.log(z))[:, 0]
    if return_lse:
        return out, lse
    return out


def softmax_row_sums(q_ae, k_vlm, k_ae) -> np.ndarray:
    """Row sums of the Eq. 1 attention probabilities, [H, Tq] (should be 1)."""
    q = np.asarray(q_ae, dtype=np.float64)
    k_all = np.concatenate([np.asarray(k_vlm, np.float64), np.asarray(k_ae, np.float64)], axis=0)
    tq, n_heads, d = q.shape
    sums = np.empty((n_heads, tq))
    for h in range(n_heads):
        s = (q[:, h, :] @ k_all[:, h, :].T) / np.sqrt(d)
        e = np.exp(s - np.max(s, axis=1, keepdims=True))
        sums[h] = np.sum(e / np.sum(e, axis=1, keepdims=True), axis=1)
    return sums


def _layer(params: dict, layer: int, name: str) -> np.ndarray:
    return np.asarray(params[name][layer], dtype=np.float64)


def expert_layers(params: dict, x: np.ndarray, k_cache, v_cache, offsets, n_heads: int, head_dim: int,
                  capture_attention: bool = False):
    """The expert's layer stack (Sec. 3.1, Eq. 1) on assembled tokens x [B, T, d].

    params: stacked over layers, matrices [out_features, in_features]:
      attn_norm [NL, d], wq/wk/wv [NL, H*D, d], wo [NL, d, H*D],
      mlp_norm [NL, d], w_gate/w_up [NL, F, d], w_down [NL, d, F].
    k_cache, v_cache: sequence of NL arrays [total_tokens, H, D]; vehicle b owns
      rows offsets[b] .. offsets[b+1]-1 of every layer. They are only read.
    Returns the residual stream after the last layer [B, T, d] and, if
    capture_attention, A [NL, B*T, H*D]: each layer's Eq. 1 output before W_o."""
    x = np.array(x, dtype=np.float64)
    offsets = np.asarray(offsets, dtype=np.int64)
    n_batch, n_tok, _ = x.shape
    n_layers = len(params["wq"])
    hd = n_heads * head_dim
    captured = np.zeros((n_layers, n_batch * n_tok, hd)) if capture_attention else None
    for layer in range(n_layers):
        wq = _layer(params, layer, "wq")
        wk = _layer(params, layer, "wk")
        wv = _layer(params, layer, "wv")
        wo = _layer(params, layer, "wo")
        wg = _layer(params, layer, "w_gate")
        wu = _layer(params, layer, "w_up")
        wd = _layer(params, layer, "w_down")
        g1 = _layer(params, layer, "attn_norm")
        g2 = _layer(params, layer, "mlp_norm")
        kc = k_cache[layer]
        vc = v_cache[layer]
        for b in range(n_batch):
            n = rms_norm(x[b], g1)
            q_ae = (n @ wq.T).reshape(n_tok, n_heads, head_dim)
            k_ae = (n @ wk.T).reshape(n_tok, n_heads, head_dim)
            v_ae = (n @ wv.T).reshape(n_tok, n_heads, head_dim)
            lo, hi = int(offsets[b]), int(offsets[b + 1])
            k_vlm = np.asarray(kc[lo:hi], dtype=np.float64)
            v_vlm = np.asarray(vc[lo:hi], dtype=np.float64)
            a = attention_eq1(q_ae, k_vlm, v_vlm, k_ae, v_ae).reshape(n_tok, hd)
            if captured is not None:
                captured[layer, b * n_tok:(b + 1) * n_tok] = a
            x[b] = x[b] + a @ wo.T
            n = rms_norm(x[b], g2)
            x[b] = x[b] + (silu(n @ wg.T) * (n @ wu.T)) @ wd.T
    return x, captured


def expert_tick(params: dict, k_cache, v_cache, offsets, frames,
                n_heads: int, head_dim: int, n_waypoints: int = 5,
                capture_attention: bool = False):
    """One expert tick for B vehicles (Sec. 3.1, Eq. 1; Sec. 3.3 deployment).

    params: dict of arrays (any float dtype; read as fp64): the layer weights of
      expert_layers plus act_emb [n_action, d], pos_emb [n_action + n_frame, d],
      final_norm [d], head_w [2, d], head_b [2].
    k_cache, v_cache, offsets: as in expert_layers.
    frames: [B, n_frame, d] frame tokens.

    Returns waypoints [B, n_waypoints, 2] (fp64) and, if capture_attention,
    also A [NL, B*T, H*D]: each layer's Eq. 1 output before W_o, token-major.
    """
    act_emb = np.asarray(params["act_emb"], np.float64)
    pos_emb = np.asarray(params["pos_emb"], np.float64)
    frames = np.asarray(frames, np.float64)
    n_batch = frames.shape[0]

    # token assembly: learned action tokens, then the frame tokens, plus the
    # learned positional embedding (expert tokens carry no rotary phase)
    x = np.concatenate([np.broadcast_to(act_emb, (n_batch,) + act_emb.shape), frames], axis=1)
    x = x + pos_emb[None, :, :]                                   # [B, T, d]
    x, captured = expert_layers(params, x, k_cache, v_cache, offsets, n_heads, head_dim, capture_attention)

    head_w = np.asarray(params["head_w"], np.float64)
    head_b = np.asarray(params["head_b"], np.float64)
    final_norm = np.asarray(params["final_norm"], np.float64)
    waypoints = rms_norm(x[:, :n_waypoints, :], final_norm) @ head_w.T + head_b
    if capture_attention:
        return waypoints, captured
    return waypoints
