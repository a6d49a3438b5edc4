"""Eq. 1 split-KV attention kernel through the C ABI (fsx_attention) against
the fp64 oracle, plus the invariants the method fixes, on ragged batches with
an empty cache, several 64-key chunks and a ragged last chunk."""
from __future__ import annotations

import math

import numpy as np
import pytest
import torch

from oracle import fsx_oracle
from paper_2607_15621_gb300 import fsx

pytestmark = pytest.mark.gpu

H, D = 32, 128


def make(lengths, n_q=42, n_own=42, cache_dtype="bf16", seed=0):
    g = torch.Generator().manual_seed(seed)
    B = len(lengths)
    off = np.concatenate([[0], np.cumsum(lengths)]).astype(np.int64)
    total = int(off[-1])
    scale = torch.exp(0.5 * torch.randn(H, D, generator=g))
    kc = torch.randn(total, H, D, generator=g) * scale
    vc = torch.randn(total, H, D, generator=g)
    if cache_dtype == "bf16":
        kc, vc = kc.to(torch.bfloat16), vc.to(torch.bfloat16)
    q = torch.randn(B * n_q, H * D, generator=g).to(torch.float16)
    ko = torch.randn(B * max(n_own, 1), H * D, generator=g).to(torch.float16)
    vo = torch.randn(B * max(n_own, 1), H * D, generator=g).to(torch.float16)
    return dict(lengths=np.asarray(lengths), off=off, kc=kc, vc=vc, q=q, ko=ko, vo=vo, n_q=n_q, n_own=n_own,
                dtype=cache_dtype, B=B)


def gpu_attention(c, n_splits):
    B, n_q, n_own = c["B"], c["n_q"], c["n_own"]
    dev = lambda t: t.to("cuda").contiguous()
    q, ko, vo, kc, vc = dev(c["q"]), dev(c["ko"]), dev(c["vo"]), dev(c["kc"]), dev(c["vc"])
    off = torch.as_tensor(c["off"], device="cuda")
    out = torch.full((B * n_q, H * D), float("nan"), device="cuda", dtype=torch.float16)
    lse = torch.empty(B, H, n_q, device="cuda", dtype=torch.float32)
    ws = torch.empty(fsx.attention_workspace_bytes(B, H, n_q, n_splits), device="cuda", dtype=torch.uint8)
    fsx.attention(q, H * D, ko, vo, H * D, n_q, n_own, kc, vc, c["dtype"], off, B, H, n_splits, out, lse, ws)
    torch.cuda.synchronize()
    return out.cpu().double().numpy(), lse.cpu().double().numpy()


def oracle_attention(c):
    outs, lses = [], []
    n_q, n_own = c["n_q"], c["n_own"]
    for b in range(c["B"]):
        lo, hi = c["off"][b], c["off"][b + 1]
        q = c["q"][b * n_q:(b + 1) * n_q].double().numpy().reshape(n_q, H, D)
        ko = c["ko"][b * n_own:(b + 1) * n_own].double().numpy().reshape(n_own, H, D)
        vo = c["vo"][b * n_own:(b + 1) * n_own].double().numpy().reshape(n_own, H, D)
        kc = c["kc"][lo:hi].double().numpy()
        vc = c["vc"][lo:hi].double().numpy()
        a, lse = fsx_oracle.attention_eq1(q, kc, vc, ko, vo, return_lse=True)
        outs.append(a.reshape(n_q, H * D))
        lses.append(lse)
    return np.concatenate(outs), np.stack(lses)


def row_err(a, b):
    return np.max(np.abs(a - b), axis=-1) / np.max(np.abs(b), axis=-1)


@pytest.mark.parametrize("cache_dtype", ["bf16", "fp32"])
@pytest.mark.parametrize("n_splits", [1, 3, 9])
def test_attention_matches_oracle(cache_dtype, n_splits):
    c = make([0, 37, 200, 65], cache_dtype=cache_dtype, seed=n_splits)
    out, lse = gpu_attention(c, n_splits)
    ref, ref_lse = oracle_attention(c)
    assert np.isfinite(out).all()
    # fp16 operands (exact for the fp16/bf16 inputs; fp32 cache rounded to fp16) with fp32 accumulation
    assert row_err(out, ref).max() < 5e-3
    assert np.max(np.abs(lse - ref_lse)) < 2e-3


def test_attention_rows_sum_to_one():
    """The GPU log-sum-exp normalises the exact scores: sum_j exp(s_j - lse) = 1."""
    c = make([150, 3], seed=11)
    _, lse = gpu_attention(c, 5)
    for b in range(c["B"]):
        lo, hi = c["off"][b], c["off"][b + 1]
        q = c["q"][b * 42:(b + 1) * 42].double().numpy().reshape(42, H, D)
        k = np.concatenate([c["kc"][lo:hi].double().numpy(),
                            c["ko"][b * 42:(b + 1) * 42].double().numpy().reshape(42, H, D)])
        s = np.einsum("qhd,khd->hqk", q, k) / math.sqrt(D)
        sums = np.exp(s - lse[b][:, :, None]).sum(-1)
        assert np.max(np.abs(sums - 1)) < 1e-3


def test_attention_permutation_invariant():
    c = make([123, 64], seed=3)
    out, _ = gpu_attention(c, 4)
    perm = np.concatenate([np.random.default_rng(0).permutation(123), 123 + np.random.default_rng(1).permutation(64)])
    c2 = dict(c, kc=c["kc"][perm], vc=c["vc"][perm])
    out2, _ = gpu_attention(c2, 4)
    assert row_err(out2, out).max() < 2e-3


def test_attention_duplicating_every_pair_invariant():
    c = make([50, 90], seed=4)
    out, _ = gpu_attention(c, 3)
    off = c["off"]
    kc = torch.cat([torch.cat([c["kc"][off[b]:off[b + 1]]] * 2) for b in range(2)])
    vc = torch.cat([torch.cat([c["vc"][off[b]:off[b + 1]]] * 2) for b in range(2)])
    ko = torch.cat([torch.cat([c["ko"][b * 42:(b + 1) * 42]] * 2) for b in range(2)])
    vo = torch.cat([torch.cat([c["vo"][b * 42:(b + 1) * 42]] * 2) for b in range(2)])
    c2 = dict(c, kc=kc, vc=vc, ko=ko, vo=vo, n_own=84, off=2 * off, lengths=2 * c["lengths"])
    out2, _ = gpu_attention(c2, 3)
    assert row_err(out2, out).max() < 2e-3


def test_attention_empty_cache_is_expert_only():
    c = make([0, 0, 0], seed=5)
    out, lse = gpu_attention(c, 2)
    ref, ref_lse = oracle_attention(c)
    assert row_err(out, ref).max() < 5e-3
    assert np.max(np.abs(lse - ref_lse)) < 2e-3


def test_attention_split_count_invariant():
    c = make([300, 1, 777], seed=6)
    base, lse1 = gpu_attention(c, 1)
    for s in (2, 7, 16, 64):
        out, lse = gpu_attention(c, s)
        assert row_err(out, base).max() < 2e-3
        assert np.max(np.abs(lse - lse1)) < 1e-3


def test_attention_small_query_counts():
    """The paper's own expert has 10 tokens; query rows beyond n_q stay untouched."""
    c = make([33, 140], n_q=10, n_own=10, seed=7)
    out, lse = gpu_attention(c, 3)
    ref, ref_lse = oracle_attention(c)
    assert row_err(out, ref).max() < 5e-3


def test_attention_bad_offsets_write_nothing():
    """Offsets beyond the caller's cache never read it: the kernels flag the
    status word and leave the output untouched (host never sees a fault)."""
    c = make([10, 20], seed=8)
    c["off"] = np.array([0, 30, 10], dtype=np.int64)  # decreasing
    B, n_q = c["B"], c["n_q"]
    off = torch.as_tensor(c["off"], device="cuda")
    out = torch.full((B * n_q, H * D), 7.0, device="cuda", dtype=torch.float16)
    ws = torch.empty(fsx.attention_workspace_bytes(B, H, n_q, 1), device="cuda", dtype=torch.uint8)
    dev = lambda t: t.to("cuda").contiguous()
    fsx.attention(dev(c["q"]), H * D, dev(c["ko"]), dev(c["vo"]), H * D, n_q, 42, dev(c["kc"]), dev(c["vc"]),
                  "bf16", off, B, H, 1, out, None, ws)
    torch.cuda.synchronize()
    # vehicle 1 (offsets 30 -> 10) must be untouched
    assert torch.all(out[n_q:] == 7.0)
    assert int(ws[:4].view(torch.int32).item()) == fsx.FSX_ERR_DEVICE_ARG
