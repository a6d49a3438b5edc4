"""Plain fp64 CPU oracle of the staleness-masked forward over a training clip.

TEST INFRASTRUCTURE, like ``fsx_oracle``: only ``tests/``, ``__graft_entry__.smoke()``
and ``bench.py``'s CPU legs may import it; it takes and returns plain numpy arrays.

What it computes (Sec. 3.2, "Staleness-Augmented Training"): at deployment the cache
the expert reads lags the current frame by up to K ticks. Training reproduces the gap:
for a staleness delta, frame j's expert block sees the backbone prefix ending at frame
j - delta, or the instruction text alone when j < delta. All frames of a clip are run
at once, and the expert blocks never see each other, so the clip forward equals one
expert tick per frame over its visible prefix. This is the forward only; the training
itself is out of scope.

Cache layout of a clip: rows 0 .. text_len-1 hold the instruction text, then every
frame f appends ``tokens_per_frame`` rows (4: the Q-Former tokens), so frame f's rows
are text_len + tokens_per_frame * f .. + tokens_per_frame - 1.

Readings where the paper is silent: "the prefix ending at frame j - delta" includes
frame j - delta's own rows; with delta = 0 a frame's block sees its own frame's
backbone rows. The expert blocks use the tick of ``fsx_oracle`` (42-token layout:
action tokens, then the frame's expert frame tokens).

Parity status: pinned in tests/test_staleness_oracle_pins.py against the per-block
attention-mask formulation the paper trains with (one torch SDPA call over all
blocks, explicit boolean mask), and closed cases.
"""
from __future__ import annotations

import numpy as np

from .fsx_oracle import expert_tick


def visible_prefix(j: int, delta: int, text_len: int, tokens_per_frame: int = 4) -> int:
    """Cache rows visible to frame j's expert block: the text, plus frames 0 .. j - delta."""
    if j < delta:
        return text_len
    return text_len + tokens_per_frame * (j - delta + 1)


def staleness_masked_forward(params: dict, k_cache, v_cache, text_len: int, frames, delta: int,
                             n_heads: int, head_dim: int, n_waypoints: int = 5, tokens_per_frame: int = 4,
                             capture_attention: bool = False):
    """Waypoints of every frame of one clip under staleness delta.

    k_cache, v_cache: NL arrays [text_len + tokens_per_frame * J, H, D], the clip's cache.
    frames: [J, n_frame, d], the expert's frame tokens of frames 0 .. J-1.
    Returns waypoints [J, n_waypoints, 2] (and, with capture_attention, every block's
    per-layer Eq. 1 outputs [J, NL, T, H*D])."""
    frames = np.asarray(frames, dtype=np.float64)
    n_frames = frames.shape[0]
    wps, atts = [], []
    for j in range(n_frames):
        p_j = visible_prefix(j, delta, text_len, tokens_per_frame)
        kc = [k[:p_j] for k in k_cache]
        vc = [v[:p_j] for v in v_cache]
        out = expert_tick(params, kc, vc, np.array([0, p_j]), frames[j:j + 1], n_heads, head_dim, n_waypoints,
                          capture_attention=capture_attention)
        if capture_attention:
            wps.append(out[0][0])
            atts.append(out[1])
        else:
            wps.append(out[0])
    if capture_attention:
        return np.stack(wps), np.stack(atts)
    return np.stack(wps)
