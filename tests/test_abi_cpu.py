"""C-ABI library checks that need no GPU: the library loads, exports every
function include/fsx.h declares, and rejects bad host arguments before any
CUDA work (status codes and messages)."""
from __future__ import annotations

import ctypes
import os
import re

import numpy as np
import pytest
import torch

from paper_2607_15621_gb300 import fsx, synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "fsx.h")


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(fsx.LIB_PATH):
        from paper_2607_15621_gb300 import build
        build.build()
    return fsx.lib()


def header_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(fsx_[a-z_0-9]+)\s*\(", text)))


def test_header_symbols_exported(lib):
    names = header_functions()
    assert len(names) >= 10
    for name in names:
        assert hasattr(lib, name), f"{name} declared in include/fsx.h but not exported"
    assert set(names) == set(fsx.declared_symbols())


def _cfg(**over):
    dims = synth.EXPERT
    cfg = fsx.make_config(dims, max_batch=4, max_total_cache_tokens=1000)
    for k, v in over.items():
        setattr(cfg, k, v)
    return cfg


def _create(lib, cfg, weights=True):
    w = synth.make_weights(synth.Dims(n_layers=1, d_model=128, n_heads=1, d_ff=64), 0) if weights else None
    keep = None
    if weights:
        wst, keep = fsx.make_weights(w)
        wp = ctypes.byref(wst)
    else:
        wp = None
    h = ctypes.c_void_p()
    st = lib.fsx_create(ctypes.byref(cfg) if cfg is not None else None, wp, 0, ctypes.byref(h))
    return st, h


def test_create_rejects_null_config(lib):
    st, h = _create(lib, None)
    assert st == fsx.FSX_ERR_INVALID_ARG
    assert "config" in fsx.last_error()
    assert not h.value


def test_create_rejects_null_weights(lib):
    st, _ = _create(lib, _cfg(), weights=False)
    assert st == fsx.FSX_ERR_INVALID_ARG


@pytest.mark.parametrize("field,value,code", [
    ("head_dim", 64, fsx.FSX_ERR_UNSUPPORTED),
    ("d_model", 500, fsx.FSX_ERR_UNSUPPORTED),
    ("d_model", 192, fsx.FSX_ERR_UNSUPPORTED),
    ("d_ff", 100, fsx.FSX_ERR_UNSUPPORTED),
    ("n_frame", 40, fsx.FSX_ERR_UNSUPPORTED),
    ("n_layers", 0, fsx.FSX_ERR_INVALID_ARG),
    ("max_batch", 0, fsx.FSX_ERR_INVALID_ARG),
    ("cache_dtype", 7, fsx.FSX_ERR_INVALID_ARG),
    ("n_waypoints", 99, fsx.FSX_ERR_INVALID_ARG),
])
def test_create_rejects_bad_shapes(lib, field, value, code):
    st, h = _create(lib, _cfg(**{field: value}))
    assert st == code, fsx.last_error()
    assert not h.value
    assert fsx.last_error()


def test_forced_allocation_failure(lib, monkeypatch):
    monkeypatch.setenv("FSX_TEST_FAIL_ALLOC", "1")
    st, h = _create(lib, _cfg(n_layers=1, d_model=128, n_heads=1, d_ff=64))
    assert st == fsx.FSX_ERR_OOM
    assert not h.value


def test_create_without_gpu_reports_cuda_error(lib):
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    st, h = _create(lib, _cfg(n_layers=1, d_model=128, n_heads=1, d_ff=64))
    assert st == fsx.FSX_ERR_CUDA
    assert not h.value


def test_tick_rejects_null_handle(lib):
    arr = (ctypes.c_void_p * 1)()
    assert lib.fsx_tick(None, arr, arr, 1, 1, 1, 1, None) == fsx.FSX_ERR_INVALID_ARG
    assert lib.fsx_tick_host(None, arr, arr, 1, 1, 1, 1, None) == fsx.FSX_ERR_INVALID_ARG
    assert lib.fsx_get_status(None, None) == fsx.FSX_ERR_INVALID_ARG
    assert lib.fsx_weight_bytes(None) == 0
    assert lib.fsx_tick_launches(None, 1) == 0
    lib.fsx_destroy(None)  # no-op


def test_attention_host_validation(lib):
    ws = fsx.attention_workspace_bytes(2, 32, 42, 12)
    assert ws == 256 + 2 * 32 * 12 * 48 * 128 * 4 + 2 * 32 * 12 * 48 * 4
    assert fsx.attention_workspace_bytes(2, 32, 42, 1) == 256
    assert fsx.attention_workspace_bytes(2, 32, 42, 8) == 256  # up to 8 splits merge on chip
    fake = 1 << 20  # never dereferenced: every case fails host validation first
    base = dict(q=fake, qs=4096 * 3, ko=fake, vo=fake, os=4096 * 3, nq=42, no=42, kc=fake, vc=fake, dt=1,
                off=fake, B=2, H=32, D=128, S=12, out=fake, lse=None, ws=fake, wsb=ws)

    def call(**kw):
        a = dict(base, **kw)
        return lib.fsx_attention(a["q"], a["qs"], a["ko"], a["vo"], a["os"], a["nq"], a["no"], a["kc"], a["vc"],
                                 a["dt"], a["off"], a["B"], a["H"], a["D"], a["S"], a["out"], a["lse"], a["ws"],
                                 a["wsb"], None)
    assert call(D=64) == fsx.FSX_ERR_UNSUPPORTED
    assert call(nq=49) == fsx.FSX_ERR_INVALID_ARG
    assert call(nq=0) == fsx.FSX_ERR_INVALID_ARG
    assert call(S=0) == fsx.FSX_ERR_INVALID_ARG
    assert call(S=65) == fsx.FSX_ERR_INVALID_ARG
    assert call(q=None) == fsx.FSX_ERR_INVALID_ARG
    assert call(wsb=ws - 1) == fsx.FSX_ERR_INVALID_ARG
    assert call(qs=4095) == fsx.FSX_ERR_INVALID_ARG
    assert call(dt=3) == fsx.FSX_ERR_INVALID_ARG
    assert "workspace" in fsx.last_error() or fsx.last_error()


# ---------------------------------------------------------------- cache append
def _append_cfg(**over):
    d = synth.BackboneDims(n_layers=1, d_model=128, n_heads=1, d_ff=64)
    cfg = fsx.AppendConfig(d.n_layers, d.d_model, d.n_heads, d.head_dim, d.d_ff, d.n_new, 4, 1000,
                           float(d.rope_base))
    for k, v in over.items():
        setattr(cfg, k, v)
    return cfg


def _append_create(lib, cfg, weights=True):
    keep = None
    if weights:
        w = synth.make_backbone_weights(synth.BackboneDims(n_layers=1, d_model=128, n_heads=1, d_ff=64), 0)
        keep = {k: np.ascontiguousarray(w[k], dtype=np.float32) for k in fsx._APPEND_WEIGHT_FIELDS}
        wst = fsx.AppendWeights(*[keep[k].ctypes.data_as(ctypes.POINTER(ctypes.c_float))
                                  for k in fsx._APPEND_WEIGHT_FIELDS])
        wp = ctypes.byref(wst)
    else:
        wp = None
    h = ctypes.c_void_p()
    st = lib.fsx_append_create(ctypes.byref(cfg) if cfg is not None else None, wp, 0, ctypes.byref(h))
    return st, h


def test_append_create_rejects_null_arguments(lib):
    st, h = _append_create(lib, None)
    assert st == fsx.FSX_ERR_INVALID_ARG and not h.value
    assert "config" in fsx.last_error()
    st, h = _append_create(lib, _append_cfg(), weights=False)
    assert st == fsx.FSX_ERR_INVALID_ARG and not h.value


@pytest.mark.parametrize("field,value,code", [
    ("head_dim", 64, fsx.FSX_ERR_UNSUPPORTED),
    ("d_model", 200, fsx.FSX_ERR_UNSUPPORTED),
    ("d_ff", 100, fsx.FSX_ERR_UNSUPPORTED),
    ("n_new", 9, fsx.FSX_ERR_UNSUPPORTED),
    ("max_batch", 65, fsx.FSX_ERR_UNSUPPORTED),
    ("n_layers", 0, fsx.FSX_ERR_INVALID_ARG),
    ("max_cache_rows", -1, fsx.FSX_ERR_INVALID_ARG),
    ("rope_base", 1.0, fsx.FSX_ERR_INVALID_ARG),
])
def test_append_create_rejects_bad_shapes(lib, field, value, code):
    st, h = _append_create(lib, _append_cfg(**{field: value}))
    assert st == code, fsx.last_error()
    assert not h.value
    assert fsx.last_error()


def test_append_create_without_gpu_reports_cuda_error(lib):
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    st, h = _append_create(lib, _append_cfg())
    assert st == fsx.FSX_ERR_CUDA and not h.value


def test_append_rejects_null_handle(lib):
    arr = (ctypes.c_void_p * 1)()
    assert lib.fsx_append(None, arr, arr, 1, 1, 1, 1, 1, None) == fsx.FSX_ERR_INVALID_ARG
    assert lib.fsx_append_get_status(None, None) == fsx.FSX_ERR_INVALID_ARG
    assert lib.fsx_append_weight_bytes(None) == 0
    lib.fsx_append_destroy(None)  # no-op
