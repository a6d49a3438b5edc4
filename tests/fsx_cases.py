"""Shared helpers of the GPU tests: seeded inputs on the device, per-vehicle
oracle runs on host copies of exactly those inputs, and tolerance checks.

Tolerances are the ones the method's parity bar fixes: every per-layer Eq. 1
output row (one token's n_heads*head_dim values at one layer) within
2e-2 * max|ref| of that row, and the waypoints within 1e-2 in relative L2.
"""
from __future__ import annotations

import functools

import numpy as np
import torch

from oracle import fsx_oracle
from paper_2607_15621_gb300 import fsx, synth

ATTN_ROW_TOL = 2e-2
WAYPOINT_TOL = 1e-2


@functools.lru_cache(maxsize=4)
def weights(dims: synth.Dims, seed: int, dtype: str):
    return synth.make_weights(dims, seed, dtype)


class Case:
    """Seeded inputs of one workload, resident on the GPU."""

    def __init__(self, dims, lengths, dtype, seed=0, gen_device="cpu"):
        self.dims = dims
        self.dtype = dtype
        self.seed = seed
        self.lengths = np.asarray(lengths, dtype=np.int64)
        self.B = len(self.lengths)
        self.w = weights(dims, seed, dtype)
        k, v, off = synth.make_cache(dims, self.lengths, seed, dtype, device=gen_device)
        self.k = [t.to("cuda") for t in k]
        self.v = [t.to("cuda") for t in v]
        self.offsets_np = off
        self.offsets = torch.as_tensor(off, device="cuda")
        self.frames = synth.make_frames(dims, self.B, seed, dtype, device=gen_device).to("cuda")
        self.total = int(off[-1])

    def expert(self, max_batch=None):
        return fsx.Expert(self.dims, self.w, max_batch or self.B, max(self.total, 1), self.dtype, self.dtype)

    def oracle_vehicle(self, b: int, capture=True):
        """Oracle tick of vehicle b alone (vehicles are independent)."""
        lo, hi = int(self.offsets_np[b]), int(self.offsets_np[b + 1])
        k = [t[lo:hi].to("cpu", torch.float32).numpy() for t in self.k]
        v = [t[lo:hi].to("cpu", torch.float32).numpy() for t in self.v]
        fr = self.frames[b:b + 1].to("cpu", torch.float64).numpy()
        d = self.dims
        return fsx_oracle.expert_tick(self.w, k, v, np.array([0, hi - lo]), fr, d.n_heads, d.head_dim,
                                      d.n_waypoints, capture_attention=capture)


def run_debug_tick(expert: fsx.Expert, case: Case):
    d = case.dims
    out = torch.empty(case.B, d.n_waypoints, 2, device="cuda", dtype=torch.float32)
    att = torch.empty(d.n_layers, case.B * d.n_tok, d.hd, device="cuda", dtype=torch.float16)
    expert.tick_debug(case.k, case.v, case.offsets, case.frames, out, att)
    torch.cuda.synchronize()
    assert expert.status() == fsx.FSX_OK
    return out.cpu().numpy().astype(np.float64), att


def run_tick(expert: fsx.Expert, case: Case):
    d = case.dims
    out = torch.empty(case.B, d.n_waypoints, 2, device="cuda", dtype=torch.float32)
    expert.tick(case.k, case.v, case.offsets, case.frames, out)
    torch.cuda.synchronize()
    assert expert.status() == fsx.FSX_OK
    return out.cpu().numpy().astype(np.float64)


def attn_row_errors(gpu_rows: np.ndarray, ref_rows: np.ndarray) -> np.ndarray:
    """max_j |gpu - ref| / max_j |ref| for every row (last axis)."""
    err = np.max(np.abs(gpu_rows - ref_rows), axis=-1)
    scale = np.max(np.abs(ref_rows), axis=-1)
    return err / np.maximum(scale, 1e-30)


def check_vehicle(case: Case, b: int, wp_gpu: np.ndarray, att_gpu: torch.Tensor, wp_tol=WAYPOINT_TOL,
                  row_tol=ATTN_ROW_TOL):
    ref_wp, ref_att = case.oracle_vehicle(b)
    T = case.dims.n_tok
    gpu_rows = att_gpu[:, b * T:(b + 1) * T].to("cpu", torch.float64).numpy()
    row_err = attn_row_errors(gpu_rows, ref_att)
    wp_err = np.linalg.norm(wp_gpu[b] - ref_wp[0]) / np.linalg.norm(ref_wp[0])
    assert row_err.max() <= row_tol, f"vehicle {b}: worst attention row error {row_err.max():.4g} > {row_tol}"
    assert wp_err <= wp_tol, f"vehicle {b}: waypoint relative L2 error {wp_err:.4g} > {wp_tol}"
    return float(row_err.max()), float(wp_err)
