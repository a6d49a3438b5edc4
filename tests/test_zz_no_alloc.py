"""fsx_attention_noalloc: the attention entry point for callers that may not
allocate device memory while running (it keeps its scratch in a static array
inside the library). Its results must equal those of fsx_attention, which
uses a caller scratch buffer, on two calls in a row with different inputs
(the second call must not see the first call's leftovers). Device-side
argument errors land in the static array's status word, which
fsx_attention_noalloc_status reads and clears."""
from __future__ import annotations

import numpy as np
import pytest
import torch

from paper_2607_15621_gb300 import fsx

pytestmark = pytest.mark.gpu

D = 128


def _inputs(lengths, seed, n_q=42, n_own=42, H=32):
    g = torch.Generator().manual_seed(seed)
    B = len(lengths)
    off = np.concatenate([[0], np.cumsum(lengths)]).astype(np.int64)
    total = int(off[-1])
    kc = (torch.randn(total, H, D, generator=g) * torch.exp(0.5 * torch.randn(H, D, generator=g))).to(torch.bfloat16)
    vc = torch.randn(total, H, D, generator=g).to(torch.bfloat16)
    q = torch.randn(B * n_q, H * D, generator=g).to(torch.float16)
    ko = torch.randn(B * n_own, H * D, generator=g).to(torch.float16)
    vo = torch.randn(B * n_own, H * D, generator=g).to(torch.float16)
    cuda = lambda t: t.to("cuda").contiguous()
    return dict(B=B, H=H, n_q=n_q, n_own=n_own, off=torch.as_tensor(off, device="cuda"), kc=cuda(kc), vc=cuda(vc),
                q=cuda(q), ko=cuda(ko), vo=cuda(vo))


def _with_buffer(c, n_splits):
    H = c["H"]
    out = torch.empty(c["B"] * c["n_q"], H * D, device="cuda", dtype=torch.float16)
    lse = torch.empty(c["B"], H, c["n_q"], device="cuda")
    ws = torch.empty(fsx.attention_workspace_bytes(c["B"], H, c["n_q"], n_splits), device="cuda", dtype=torch.uint8)
    fsx.attention(c["q"], H * D, c["ko"], c["vo"], H * D, c["n_q"], c["n_own"], c["kc"], c["vc"], "bf16", c["off"],
                  c["B"], H, n_splits, out, lse, ws)
    return out, lse


def _no_alloc(c, n_splits):
    H = c["H"]
    out = torch.full((c["B"] * c["n_q"], H * D), float("nan"), device="cuda", dtype=torch.float16)
    lse = torch.full((c["B"], H, c["n_q"]), float("nan"), device="cuda")
    fsx.attention_noalloc(c["q"], H * D, c["ko"], c["vo"], H * D, c["n_q"], c["n_own"], c["kc"], c["vc"], "bf16",
                          c["off"], c["B"], H, n_splits, out, lse)
    return out, lse


def _row_err(a, b):
    a = a.double().cpu().numpy()
    b = b.double().cpu().numpy()
    return np.max(np.abs(a - b), axis=-1) / np.max(np.abs(b), axis=-1)


def test_no_alloc_matches_buffered_entry_on_consecutive_calls():
    # 16 splits of 8 heads keep per-split partials in the static scratch (more than
    # 8 splits are merged through it); 5 and 1 splits use only its status word
    cases = [(_inputs([200], seed=1, H=8), 16), (_inputs([129, 0], seed=2), 5), (_inputs([0, 37, 300], seed=4), 1)]
    for c, n_splits in cases:  # calls in a row; each overwrites the shared scratch
        ref_out, ref_lse = _with_buffer(c, n_splits)
        out, lse = _no_alloc(c, n_splits)
        torch.cuda.synchronize()
        assert torch.isfinite(out.float()).all() and torch.isfinite(lse).all()
        assert _row_err(out, ref_out).max() < 2e-3
        assert torch.max(torch.abs(lse - ref_lse)).item() < 1e-3


def test_no_alloc_rejects_requests_beyond_its_scratch():
    c = _inputs([10], seed=3)
    H = c["H"]
    out = torch.empty(c["B"] * c["n_q"], H * D, device="cuda", dtype=torch.float16)
    too_many = 64  # 32 heads x 64 splits x 24.8 KB > 4 MiB
    with pytest.raises(fsx.FsxError) as e:
        fsx.attention_noalloc(c["q"], H * D, c["ko"], c["vo"], H * D, c["n_q"], c["n_own"], c["kc"], c["vc"],
                              "bf16", c["off"], c["B"], H, too_many, out, None)
    assert e.value.status == fsx.FSX_ERR_INVALID_ARG
    assert "scratch" in str(e.value)


def test_no_alloc_reports_device_side_offset_errors_through_its_status_word():
    c = _inputs([50, 30], seed=5)
    H = c["H"]
    assert fsx.attention_noalloc_status() == fsx.FSX_OK  # nothing pending from earlier calls
    # offsets [0, 50, 20]: vehicle 1's range runs backwards; its rows must stay untouched
    bad = torch.as_tensor(np.array([0, 50, 20], dtype=np.int64), device="cuda")
    out = torch.full((c["B"] * c["n_q"], H * D), float("nan"), device="cuda", dtype=torch.float16)
    fsx.attention_noalloc(c["q"], H * D, c["ko"], c["vo"], H * D, c["n_q"], c["n_own"], c["kc"], c["vc"], "bf16",
                          bad, c["B"], H, 1, out, None)
    assert fsx.attention_noalloc_status() == fsx.FSX_ERR_DEVICE_ARG
    assert torch.isnan(out[c["n_q"]:].float()).all()
    assert fsx.attention_noalloc_status() == fsx.FSX_OK  # read-and-clear
    # a negative first offset with one vehicle: nothing is written at all
    neg = torch.as_tensor(np.array([-4, 20], dtype=np.int64), device="cuda")
    out1 = torch.full((c["n_q"], H * D), float("nan"), device="cuda", dtype=torch.float16)
    fsx.attention_noalloc(c["q"], H * D, c["ko"], c["vo"], H * D, c["n_q"], c["n_own"], c["kc"], c["vc"], "bf16",
                          neg, 1, H, 1, out1, None)
    assert fsx.attention_noalloc_status() == fsx.FSX_ERR_DEVICE_ARG
    assert torch.isnan(out1.float()).all()
    # the next good call runs normally and leaves the word clear
    ref_out, _ = _with_buffer(c, 5)
    out2, _ = _no_alloc(c, 5)
    assert fsx.attention_noalloc_status() == fsx.FSX_OK
    assert _row_err(out2, ref_out).max() < 2e-3
