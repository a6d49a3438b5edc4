"""Plain fp64 CPU oracle of the expert tick with the paper's own token layout.

TEST INFRASTRUCTURE, like ``fsx_oracle``: only ``tests/``, ``__graft_entry__.smoke()``
and ``bench.py``'s CPU legs may import it; it takes and returns plain numpy arrays and
imports nothing from the product path.

What it computes (Sec. 3.1): per frame the expert consumes ten tokens -- one state
token embedding the previous predicted waypoints, the previous control triplet, the
current speed and the target point; the current frame's four visual tokens; and five
learnable waypoint queries -- and a two-layer head decodes the five query outputs to
five (x, y) waypoints. The layer stack between them is the same as in ``fsx_oracle``
(Eq. 1 attention over [cache ; own keys], output projection, SwiGLU block).

  s_b      = [w_prev (5 x 2), (throttle, steer, brake), speed, target (x, y)]   16 values
  t_state  = W_s2 silu(W_s1 s_b + b_s1) + b_s2                                  (state MLP)
  X_b      = [t_state ; V_b (4 visual tokens) ; E_q (5 queries)] + P_pos
  X_b      = expert_layers(X_b)
  w_i      = W_h2 silu(W_h1 RMSNorm(X_{b, 5+i}; g_f) + b_h1) + b_h2,  i = 0..4   (two-layer head)

Readings where the paper is silent:
  * the 16 state values in the order above (the paper lists the four quantities);
  * both MLPs: two Linear layers with bias and a SiLU between them, hidden width d
    (the activation of the expert's feed-forward blocks);
  * the head reads the final-RMSNorm output of each query token, as the single-layer
    head of ``fsx_oracle`` does;
  * visual tokens arrive at width d (the Q-Former pipeline is out of scope).

Parity status: pinned in tests/test_paper_tokens_oracle_pins.py against a torch
composition, closed forms with zeroed branches, a hand-derived case and invariants.
"""
from __future__ import annotations

import numpy as np

from .fsx_oracle import expert_layers, rms_norm, silu

STATE_DIM = 16
N_VISUAL = 4
N_QUERY = 5


def state_token(params: dict, state: np.ndarray) -> np.ndarray:
    """State MLP: [B, 16] ego state -> [B, d] state token."""
    s = np.asarray(state, dtype=np.float64)
    h = silu(s @ np.asarray(params["state_w1"], np.float64).T + np.asarray(params["state_b1"], np.float64))
    return h @ np.asarray(params["state_w2"], np.float64).T + np.asarray(params["state_b2"], np.float64)


def waypoint_head(params: dict, q_tokens: np.ndarray) -> np.ndarray:
    """Two-layer head on the query tokens' final states [B, 5, d] -> waypoints [B, 5, 2]."""
    n = rms_norm(q_tokens, np.asarray(params["final_norm"], np.float64))
    h = silu(n @ np.asarray(params["head_w1"], np.float64).T + np.asarray(params["head_b1"], np.float64))
    return h @ np.asarray(params["head_w2"], np.float64).T + np.asarray(params["head_b2"], np.float64)


def expert_tick_paper_tokens(params: dict, k_cache, v_cache, offsets, visual, state,
                             n_heads: int, head_dim: int, capture_attention: bool = False):
    """One expert tick for B vehicles with the ten-token layout.

    params: the layer weights of ``fsx_oracle.expert_layers`` plus
      state_w1 [d, 16], state_b1 [d], state_w2 [d, d], state_b2 [d],
      query_emb [5, d], pos_emb [10, d], final_norm [d],
      head_w1 [d, d], head_b1 [d], head_w2 [2, d], head_b2 [2].
    k_cache, v_cache, offsets: as in ``fsx_oracle.expert_layers`` (read only).
    visual: [B, 4, d] the current frame's visual tokens.  state: [B, 16].
    Returns waypoints [B, 5, 2] and, if capture_attention, each layer's Eq. 1 output
    [NL, B*10, H*D]."""
    visual = np.asarray(visual, dtype=np.float64)
    n_batch = visual.shape[0]
    t_state = state_token(params, state)                                      # [B, d]
    queries = np.asarray(params["query_emb"], np.float64)
    x = np.concatenate([t_state[:, None, :], visual,
                        np.broadcast_to(queries, (n_batch,) + queries.shape)], axis=1)
    x = x + np.asarray(params["pos_emb"], np.float64)[None, :, :]             # [B, 10, d]
    x, captured = expert_layers(params, x, k_cache, v_cache, offsets, n_heads, head_dim, capture_attention)
    waypoints = waypoint_head(params, x[:, 1 + N_VISUAL:, :])
    if capture_attention:
        return waypoints, captured
    return waypoints
