"""Incremental cache append (fsx_append, Sec. 1 and Sec. 3.3) through the C ABI
against the fp64 append oracle on the same seeded inputs, at the full backbone
width with two layers.

Tolerance: the method states none for the append, so it takes the bar of the
tick's attention rows. Every row -- one token's hidden state (d values), or one
appended cache row (n_heads * head_dim values) -- has max |err| <= 2e-2 * max
|ref| of that row. The arithmetic behind it is as follows. Weights are stored
fp16 (exact for the bf16-valued synthetic weights). The GEMM operands are fp16,
about 2^-11 relative each. The appended rows are rounded to bf16, 2^-9 relative.
Everything else is fp32. Over two layers that gives errors of a few 1e-3 of a
row's largest entry.
"""
from __future__ import annotations

import functools

import numpy as np
import pytest
import torch

from oracle import append_oracle
from paper_2607_15621_gb300 import fsx, synth

pytestmark = pytest.mark.gpu

DIMS = synth.BackboneDims(n_layers=2)
ROW_TOL = 2e-2
H, D, HD = DIMS.n_heads, DIMS.head_dim, DIMS.hd


@functools.lru_cache(maxsize=1)
def weights():
    return synth.make_backbone_weights(DIMS, 0, "bf16")


def row_err(got, ref):
    got = np.asarray(got, np.float64).reshape(-1, np.shape(ref)[-1])
    ref = np.asarray(ref, np.float64).reshape(got.shape)
    return np.max(np.abs(got - ref), axis=-1) / np.maximum(np.max(np.abs(ref), axis=-1), 1e-30)


def run(ap, kc, vc, offsets, dst, x):
    hidden = torch.empty(x.shape[0], DIMS.n_new, DIMS.d_model, device="cuda", dtype=torch.float32)
    ap.append(kc, vc, torch.as_tensor(offsets, device="cuda"), torch.as_tensor(dst, device="cuda"), x, hidden)
    torch.cuda.synchronize()
    assert ap.status() == fsx.FSX_OK
    return hidden.cpu().numpy()


def test_append_matches_oracle_ragged():
    """Three vehicles with 0, 37 and 130 cached tokens, one call."""
    lengths = [0, 37, 130]
    B, n = len(lengths), DIMS.n_new
    off = np.concatenate([[0], np.cumsum(lengths)]).astype(np.int64)
    total = int(off[-1])
    dst = np.array([total + n * b for b in range(B)], dtype=np.int64)
    rows = total + n * B + 5
    g = torch.Generator().manual_seed(3)
    kc = [(torch.randn(rows, H, D, generator=g) * torch.exp(0.5 * torch.randn(H, D, generator=g)))
          .to(torch.bfloat16).cuda() for _ in range(DIMS.n_layers)]
    vc = [torch.randn(rows, H, D, generator=g).to(torch.bfloat16).cuda() for _ in range(DIMS.n_layers)]
    before = [t.clone() for t in kc + vc]
    x = synth.make_append_tokens(DIMS, B, seed=4).cuda()
    ap = fsx.Append(DIMS, weights(), max_batch=4, max_cache_rows=rows)
    try:
        hidden = run(ap, kc, vc, off, dst, x)
    finally:
        ap.close()
    h_ref, k_ref, v_ref = append_oracle.backbone_append(
        weights(), [t[:total].float().cpu().numpy() for t in kc], [t[:total].float().cpu().numpy() for t in vc],
        off, x.float().cpu().numpy(), H, D)
    assert np.isfinite(hidden).all()
    assert row_err(hidden, h_ref).max() <= ROW_TOL
    written = np.concatenate([np.arange(d0, d0 + n) for d0 in dst])
    for l in range(DIMS.n_layers):
        assert row_err(kc[l][written].float().cpu().numpy(), k_ref[l]).max() <= ROW_TOL
        assert row_err(vc[l][written].float().cpu().numpy(), v_ref[l]).max() <= ROW_TOL
    keep = np.setdiff1d(np.arange(rows), written)
    for t0, t1 in zip(before, kc + vc):  # every other row is untouched
        assert torch.equal(t0[keep].view(torch.int16), t1[keep].view(torch.int16))


def test_append_equals_monolithic_forward():
    """The paper's golden equivalence on the GPU: a cache built from empty, four
    tokens per call, holds the rows of the monolithic forward over the whole
    sequence, and the last call's hidden states are that forward's last rows."""
    n, calls = DIMS.n_new, 5
    S = n * calls
    kc = [torch.zeros(S, H, D, dtype=torch.bfloat16, device="cuda") for _ in range(DIMS.n_layers)]
    vc = [torch.zeros(S, H, D, dtype=torch.bfloat16, device="cuda") for _ in range(DIMS.n_layers)]
    x_all = synth.make_append_tokens(DIMS, calls, seed=9).cuda()
    ap = fsx.Append(DIMS, weights(), max_batch=1, max_cache_rows=S)
    try:
        for c in range(calls):
            hidden = run(ap, kc, vc, np.array([0, n * c]), np.array([n * c]), x_all[c:c + 1])
    finally:
        ap.close()
    h_full, k_full, v_full = append_oracle.backbone_prefill(weights(), x_all.float().cpu().numpy().reshape(S, -1),
                                                            H, D)
    for l in range(DIMS.n_layers):
        assert row_err(kc[l].float().cpu().numpy(), k_full[l]).max() <= ROW_TOL
        assert row_err(vc[l].float().cpu().numpy(), v_full[l]).max() <= ROW_TOL
    assert row_err(hidden, h_full[S - n:]).max() <= ROW_TOL


def test_append_device_check_rejects_bad_destinations():
    """Destination rows that overlap cached rows or run past the buffer set the
    status word, and the call writes no cache row; a valid call then succeeds."""
    rows, n = 64, DIMS.n_new
    kc = [torch.randn(rows, H, D, device="cuda").to(torch.bfloat16) for _ in range(DIMS.n_layers)]
    vc = [torch.randn(rows, H, D, device="cuda").to(torch.bfloat16) for _ in range(DIMS.n_layers)]
    before = [t.clone() for t in kc + vc]
    x = synth.make_append_tokens(DIMS, 1, seed=5).cuda()
    ap = fsx.Append(DIMS, weights(), max_batch=2, max_cache_rows=rows)
    try:
        hidden = torch.empty(1, n, DIMS.d_model, device="cuda")
        for off, dst in (([0, 10], [5]), ([0, 10], [rows - 2]), ([0, 70], [0])):
            ap.append(kc, vc, torch.tensor(off, device="cuda"), torch.tensor(dst, device="cuda"), x, hidden)
            assert ap.status() == fsx.FSX_ERR_DEVICE_ARG
            for t0, t1 in zip(before, kc + vc):
                assert torch.equal(t0.view(torch.int16), t1.view(torch.int16))
        x2 = synth.make_append_tokens(DIMS, 2, seed=6).cuda()
        h2 = torch.empty(2, n, DIMS.d_model, device="cuda")
        ap.append(kc, vc, torch.tensor([0, 3, 5], device="cuda"), torch.tensor([20, 22], device="cuda"), x2, h2)
        assert ap.status() == fsx.FSX_ERR_DEVICE_ARG  # the two destination ranges overlap
        out = run(ap, kc, vc, np.array([0, 10]), np.array([10]), x)
        assert np.isfinite(out).all()
    finally:
        ap.close()


def test_append_host_argument_errors():
    rows = 16
    kc = [torch.zeros(rows, H, D, dtype=torch.bfloat16, device="cuda") for _ in range(DIMS.n_layers)]
    x = synth.make_append_tokens(DIMS, 2, seed=7).cuda()
    hidden = torch.empty(2, DIMS.n_new, DIMS.d_model, device="cuda")
    off = torch.tensor([0, 0, 0], device="cuda")
    dst = torch.tensor([0, 4], device="cuda")
    ap = fsx.Append(DIMS, weights(), max_batch=1, max_cache_rows=rows)
    try:
        with pytest.raises(fsx.FsxError) as e:
            ap.append(kc, kc, off, dst, x, hidden)  # B = 2 > max_batch = 1
        assert e.value.status == fsx.FSX_ERR_INVALID_ARG
        with pytest.raises(fsx.FsxError):
            ap.append(kc[:-1] + [None], kc, off, dst, x[:1], hidden)
        with pytest.raises(fsx.FsxError):
            ap.append(kc, kc, off, None, x[:1], hidden)
    finally:
        ap.close()


@pytest.mark.parametrize("concurrent", [False, True])
def test_append_full_depth_one_vehicle(concurrent):
    """All 32 layers of the backbone, one vehicle with the paper-shaped 224 cached tokens
    (64 instruction + 40 frames x 4): the depth the bench runs, where bf16 rounding of the
    written rows compounds over the layers. Both GEMM schedules (split K, and the one of the
    concurrent fast-slow session without it)."""
    dims = synth.BackboneDims()
    w = synth.make_backbone_weights(dims, 1, "bf16")
    L, n = 224, dims.n_new
    k0, v0, _ = synth.make_cache(synth.Dims(n_layers=dims.n_layers), [L], 1, "bf16")
    rows = L + n
    kc = [torch.zeros(rows, H, D, dtype=torch.bfloat16, device="cuda") for _ in range(dims.n_layers)]
    vc = [torch.zeros(rows, H, D, dtype=torch.bfloat16, device="cuda") for _ in range(dims.n_layers)]
    for dst_t, src in zip(kc + vc, k0 + v0):
        dst_t[:L] = src.cuda()
    x = synth.make_append_tokens(dims, 1, seed=2).cuda()
    ap = fsx.Append(dims, w, max_batch=1, max_cache_rows=rows)
    try:
        fsx.lib().fsx_append_set_concurrent(ap.h, 1 if concurrent else 0)
        hidden = torch.empty(1, n, dims.d_model, device="cuda")
        ap.append(kc, vc, torch.tensor([0, L], device="cuda"), torch.tensor([L], device="cuda"), x, hidden)
        torch.cuda.synchronize()
        assert ap.status() == fsx.FSX_OK
        hidden = hidden.cpu().numpy()
    finally:
        ap.close()
    h_ref, k_ref, v_ref = append_oracle.backbone_append(w, [t.float().numpy() for t in k0], [t.float().numpy() for t in v0],
                                                        np.array([0, L]), x.float().cpu().numpy(), H, D)
    assert row_err(hidden, h_ref).max() <= ROW_TOL
    for l in range(dims.n_layers):
        assert row_err(kc[l][L:].float().cpu().numpy(), k_ref[l]).max() <= ROW_TOL, l
        assert row_err(vc[l][L:].float().cpu().numpy(), v_ref[l]).max() <= ROW_TOL, l
