"""Thin ctypes binding of libfsx.so (include/fsx.h): argument marshalling only.

Every step of the tick runs in the library's CUDA kernels; this module only
turns torch tensors / numpy arrays into pointers, sizes and a cudaStream_t.
Importing it fails loudly when the compiled library is missing.
"""
from __future__ import annotations

import ctypes
import os
from typing import Sequence

import numpy as np

from .synth import Dims

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "_lib", "libfsx.so")

FSX_OK = 0
FSX_ERR_INVALID_ARG = 1
FSX_ERR_UNSUPPORTED = 2
FSX_ERR_OOM = 3
FSX_ERR_CUDA = 4
FSX_ERR_TIMEOUT = 5
FSX_ERR_DEVICE_ARG = 6
FSX_ERR_RANGE = 7
FSX_F32 = 0
FSX_BF16 = 1
FSX_SCHED_SERIAL = 0
FSX_SCHED_CONCURRENT = 1

KCLASS = {"qkv": 0, "attention": 1, "out_proj": 2, "gate_up": 3, "down": 4, "persistent": 5}


class FsxError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"fsx status {status}: {message}")
        self.status = status


class Config(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int), ("d_model", ctypes.c_int), ("n_heads", ctypes.c_int),
                ("head_dim", ctypes.c_int), ("d_ff", ctypes.c_int), ("n_action", ctypes.c_int),
                ("n_frame", ctypes.c_int), ("n_waypoints", ctypes.c_int), ("max_batch", ctypes.c_int),
                ("max_total_cache_tokens", ctypes.c_longlong), ("cache_dtype", ctypes.c_int),
                ("frame_dtype", ctypes.c_int)]


_WEIGHT_FIELDS = ["act_emb", "pos_emb", "attn_norm", "wq", "wk", "wv", "wo", "mlp_norm", "w_gate",
                  "w_up", "w_down", "final_norm", "head_w", "head_b"]


class Weights(ctypes.Structure):
    _fields_ = [(name, ctypes.POINTER(ctypes.c_float)) for name in _WEIGHT_FIELDS]


_PAPER_WEIGHT_FIELDS = ["state_w1", "state_b1", "state_w2", "state_b2", "query_emb", "pos_emb", "attn_norm", "wq",
                        "wk", "wv", "wo", "mlp_norm", "w_gate", "w_up", "w_down", "final_norm", "head_w1", "head_b1",
                        "head_w2", "head_b2"]


class PaperWeights(ctypes.Structure):
    _fields_ = [(name, ctypes.POINTER(ctypes.c_float)) for name in _PAPER_WEIGHT_FIELDS]


class AppendConfig(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int), ("d_model", ctypes.c_int), ("n_heads", ctypes.c_int),
                ("head_dim", ctypes.c_int), ("d_ff", ctypes.c_int), ("n_new", ctypes.c_int),
                ("max_batch", ctypes.c_int), ("max_cache_rows", ctypes.c_longlong), ("rope_base", ctypes.c_float)]


_APPEND_WEIGHT_FIELDS = ["attn_norm", "wq", "wk", "wv", "wo", "mlp_norm", "w_gate", "w_up", "w_down"]


class AppendWeights(ctypes.Structure):
    _fields_ = [(name, ctypes.POINTER(ctypes.c_float)) for name in _APPEND_WEIGHT_FIELDS]


def _load():
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is missing: build it with paper_2607_15621_gb300.build.build()")
    lib = ctypes.CDLL(LIB_PATH)
    vp, i32, i64p = ctypes.c_void_p, ctypes.c_int, ctypes.POINTER(ctypes.c_int64)
    vpp = ctypes.POINTER(ctypes.c_void_p)
    fp = ctypes.POINTER(ctypes.c_float)
    sig = {
        "fsx_create": (i32, [ctypes.POINTER(Config), ctypes.POINTER(Weights), i32, ctypes.POINTER(vp)]),
        "fsx_tick": (i32, [vp, vpp, vpp, vp, i32, vp, vp, vp]),
        "fsx_tick_host": (i32, [vp, vpp, vpp, vp, i32, vp, vp, vp]),
        "fsx_tick_debug": (i32, [vp, vpp, vpp, vp, i32, vp, vp, vp, vp]),
        "fsx_tick_ranges": (i32, [vp, vpp, vpp, vp, vp, i32, vp, vp, vp]),
        "fsx_tick_ranges_debug": (i32, [vp, vpp, vpp, vp, vp, i32, vp, vp, vp, vp]),
        "fsx_get_status": (i32, [vp, vp]),
        "fsx_last_error": (ctypes.c_char_p, []),
        "fsx_destroy": (None, [vp]),
        "fsx_set_wait_limit": (i32, [vp, ctypes.c_ulonglong]),
        "fsx_weight_bytes": (ctypes.c_longlong, [vp]),
        "fsx_tick_launches": (i32, [vp, i32]),
        "fsx_set_kernel_timing": (i32, [vp, i32, i32]),
        "fsx_kernel_time": (i32, [vp, fp, ctypes.POINTER(ctypes.c_int)]),
        "fsx_attention_workspace_bytes": (ctypes.c_size_t, [i32, i32, i32, i32]),
        "fsx_attention": (i32, [vp, ctypes.c_longlong, vp, vp, ctypes.c_longlong, i32, i32, vp, vp, i32,
                                vp, i32, i32, i32, i32, vp, vp, vp, ctypes.c_size_t, vp]),
        "fsx_attention_noalloc": (i32, [vp, ctypes.c_longlong, vp, vp, ctypes.c_longlong, i32, i32, vp, vp,
                                        i32, vp, i32, i32, i32, i32, vp, vp, vp]),
        "fsx_attention_noalloc_status": (i32, [vp]),
        "fsx_paper_create": (i32, [ctypes.POINTER(Config), ctypes.POINTER(PaperWeights), i32, ctypes.POINTER(vp)]),
        "fsx_paper_tick": (i32, [vp, vpp, vpp, vp, i32, vp, vp, vp, vp]),
        "fsx_append_set_concurrent": (i32, [vp, i32]),
        "fsx_session_create": (i32, [vp, vp, vpp, vpp, i32, i32, ctypes.c_longlong, ctypes.c_longlong, i32, i32,
                                     ctypes.POINTER(vp)]),
        "fsx_session_append": (i32, [vp, vp, vp]),
        "fsx_session_tick": (i32, [vp, vp, vp, ctypes.POINTER(ctypes.c_longlong)]),
        "fsx_session_committed": (ctypes.c_longlong, [vp]),
        "fsx_session_reserved": (ctypes.c_longlong, [vp]),
        "fsx_session_tick_stream": (vp, [vp]),
        "fsx_session_append_stream": (vp, [vp]),
        "fsx_session_sync": (i32, [vp]),
        "fsx_session_destroy": (None, [vp]),
        "fsx_append_create": (i32, [ctypes.POINTER(AppendConfig), ctypes.POINTER(AppendWeights), i32,
                                    ctypes.POINTER(vp)]),
        "fsx_append": (i32, [vp, vpp, vpp, vp, vp, i32, vp, vp, vp]),
        "fsx_append_get_status": (i32, [vp, vp]),
        "fsx_append_weight_bytes": (ctypes.c_longlong, [vp]),
        "fsx_append_destroy": (None, [vp]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    return lib


_lib = None


def lib():
    global _lib
    if _lib is None:
        _lib = _load()
    return _lib


def declared_symbols() -> list[str]:
    return ["fsx_create", "fsx_tick", "fsx_tick_host", "fsx_tick_debug", "fsx_tick_ranges", "fsx_tick_ranges_debug",
            "fsx_get_status", "fsx_last_error",
            "fsx_destroy", "fsx_weight_bytes", "fsx_tick_launches", "fsx_set_kernel_timing",
            "fsx_kernel_time", "fsx_attention_workspace_bytes", "fsx_attention", "fsx_attention_noalloc",
            "fsx_attention_noalloc_status", "fsx_paper_create", "fsx_paper_tick", "fsx_append_create", "fsx_append",
            "fsx_append_get_status", "fsx_append_weight_bytes", "fsx_append_destroy", "fsx_append_set_concurrent",
            "fsx_session_create", "fsx_session_append", "fsx_session_tick", "fsx_session_committed",
            "fsx_session_reserved", "fsx_session_tick_stream", "fsx_session_append_stream", "fsx_session_sync",
            "fsx_session_destroy", "fsx_set_wait_limit"]


def last_error() -> str:
    return lib().fsx_last_error().decode()


def check(status: int):
    if status != FSX_OK:
        raise FsxError(status, last_error())


def _ptr(t) -> int:
    """Device or host address of a torch tensor / numpy array (None -> 0)."""
    if t is None:
        return 0
    if isinstance(t, np.ndarray):
        return t.ctypes.data
    return t.data_ptr()


def _stream(stream) -> int:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _ptr_array(tensors: Sequence) -> ctypes.Array:
    arr = (ctypes.c_void_p * len(tensors))()
    for i, t in enumerate(tensors):
        arr[i] = _ptr(t)
    return arr


def make_config(dims: Dims, max_batch: int, max_total_cache_tokens: int, cache_dtype: str = "bf16",
                frame_dtype: str = "bf16") -> Config:
    code = {"fp32": FSX_F32, "bf16": FSX_BF16}
    return Config(dims.n_layers, dims.d_model, dims.n_heads, dims.head_dim, dims.d_ff, dims.n_action,
                  dims.n_frame, dims.n_waypoints, max_batch, max_total_cache_tokens,
                  code[cache_dtype], code[frame_dtype])


def make_weights(weights: dict):
    """ctypes struct of host fp32 pointers plus the contiguous arrays it points to."""
    keep = {k: np.ascontiguousarray(weights[k], dtype=np.float32) for k in _WEIGHT_FIELDS}
    st = Weights(*[keep[k].ctypes.data_as(ctypes.POINTER(ctypes.c_float)) for k in _WEIGHT_FIELDS])
    return st, keep


class Expert:
    """Owns one fsx handle (weights uploaded at construction)."""

    def __init__(self, dims: Dims, weights: dict, max_batch: int, max_total_cache_tokens: int,
                 cache_dtype: str = "bf16", frame_dtype: str = "bf16", device: int = 0):
        self.dims = dims
        self.cfg = make_config(dims, max_batch, max_total_cache_tokens, cache_dtype, frame_dtype)
        wst, keep = make_weights(weights)
        h = ctypes.c_void_p()
        check(lib().fsx_create(ctypes.byref(self.cfg), ctypes.byref(wst), device, ctypes.byref(h)))
        self.h = h
        del keep

    def close(self):
        if getattr(self, "h", None) and self.h.value:
            lib().fsx_destroy(self.h)
            self.h = ctypes.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def tick(self, k_layers, v_layers, offsets, frames, out, stream=None, starts=None):
        """One tick; with `starts`, vehicle b reads rows starts[b] .. starts[b] + L_b - 1."""
        B = int(frames.shape[0])
        if starts is None:
            check(lib().fsx_tick(self.h, _ptr_array(k_layers), _ptr_array(v_layers), _ptr(offsets), B,
                                 _ptr(frames), _ptr(out), _stream(stream)))
        else:
            check(lib().fsx_tick_ranges(self.h, _ptr_array(k_layers), _ptr_array(v_layers), _ptr(starts),
                                        _ptr(offsets), B, _ptr(frames), _ptr(out), _stream(stream)))
        return out

    def tick_host(self, k_layers, v_layers, offsets_host: np.ndarray, frames_host, out_host: np.ndarray,
                  stream=None):
        B = int(frames_host.shape[0])
        check(lib().fsx_tick_host(self.h, _ptr_array(k_layers), _ptr_array(v_layers), _ptr(offsets_host), B,
                                  _ptr(frames_host), _ptr(out_host), _stream(stream)))
        return out_host

    def tick_debug(self, k_layers, v_layers, offsets, frames, out, attn_out, stream=None, starts=None):
        B = int(frames.shape[0])
        if starts is None:
            check(lib().fsx_tick_debug(self.h, _ptr_array(k_layers), _ptr_array(v_layers), _ptr(offsets), B,
                                       _ptr(frames), _ptr(out), _ptr(attn_out), _stream(stream)))
        else:
            check(lib().fsx_tick_ranges_debug(self.h, _ptr_array(k_layers), _ptr_array(v_layers), _ptr(starts),
                                              _ptr(offsets), B, _ptr(frames), _ptr(out), _ptr(attn_out),
                                              _stream(stream)))
        return out, attn_out

    def status(self, stream=None) -> int:
        return lib().fsx_get_status(self.h, _stream(stream))

    def weight_bytes(self) -> int:
        return int(lib().fsx_weight_bytes(self.h))

    def set_wait_limit(self, ns: int):
        """Test hook: limit of the single-launch tick's device-wide waits (0 = the default 1 s)."""
        check(lib().fsx_set_wait_limit(self.h, ns))

    def launches(self, B: int) -> int:
        return int(lib().fsx_tick_launches(self.h, B))

    def set_kernel_timing(self, enable: bool, kclass: str = "qkv"):
        check(lib().fsx_set_kernel_timing(self.h, int(enable), KCLASS[kclass]))

    def kernel_time(self):
        ms = ctypes.c_float()
        n = ctypes.c_int()
        check(lib().fsx_kernel_time(self.h, ctypes.byref(ms), ctypes.byref(n)))
        return float(ms.value), int(n.value)


class PaperExpert(Expert):
    """A tick handle of the paper's ten-token layout (fsx_paper_create / fsx_paper_tick):
    state token, four visual tokens, five waypoint queries and a two-layer head over the
    same layer stack. Argument marshalling only."""

    def __init__(self, dims: Dims, weights: dict, max_batch: int, max_total_cache_tokens: int,
                 cache_dtype: str = "bf16", visual_dtype: str = "bf16", device: int = 0):
        self.dims = dims
        self.cfg = make_config(dims, max_batch, max_total_cache_tokens, cache_dtype, visual_dtype)
        keep = {k: np.ascontiguousarray(weights[k], dtype=np.float32) for k in _PAPER_WEIGHT_FIELDS}
        wst = PaperWeights(*[keep[k].ctypes.data_as(ctypes.POINTER(ctypes.c_float)) for k in _PAPER_WEIGHT_FIELDS])
        h = ctypes.c_void_p()
        check(lib().fsx_paper_create(ctypes.byref(self.cfg), ctypes.byref(wst), device, ctypes.byref(h)))
        self.h = h
        del keep

    def paper_tick(self, k_layers, v_layers, offsets, visual, state, out, stream=None):
        B = int(visual.shape[0])
        check(lib().fsx_paper_tick(self.h, _ptr_array(k_layers), _ptr_array(v_layers), _ptr(offsets), B,
                                   _ptr(visual), _ptr(state), _ptr(out), _stream(stream)))
        return out


def attention_workspace_bytes(B: int, n_heads: int, n_q: int, n_splits: int) -> int:
    return int(lib().fsx_attention_workspace_bytes(B, n_heads, n_q, n_splits))


def attention(q, q_stride, k_own, v_own, own_stride, n_q, n_own, k_cache, v_cache, cache_dtype, offsets, B,
              n_heads, n_splits, out, lse, workspace, stream=None):
    """Eq. 1 alone through the C ABI (fp16 tensors, int64 offsets, caller scratch)."""
    code = {"fp32": FSX_F32, "bf16": FSX_BF16}[cache_dtype]
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    check(lib().fsx_attention(_ptr(q), q_stride, _ptr(k_own), _ptr(v_own), own_stride, n_q, n_own,
                              _ptr(k_cache), _ptr(v_cache), code, _ptr(offsets), B, n_heads, 128, n_splits,
                              _ptr(out), _ptr(lse), _ptr(workspace), ws_bytes, _stream(stream)))
    return out


def attention_noalloc(q, q_stride, k_own, v_own, own_stride, n_q, n_own, k_cache, v_cache, cache_dtype, offsets,
                      B, n_heads, n_splits, out, lse, stream=None):
    """fsx_attention_noalloc through the C ABI: same results as attention(), with the
    library's static scratch instead of a caller buffer (nothing is allocated)."""
    code = {"fp32": FSX_F32, "bf16": FSX_BF16}[cache_dtype]
    check(lib().fsx_attention_noalloc(_ptr(q), q_stride, _ptr(k_own), _ptr(v_own), own_stride, n_q, n_own,
                                      _ptr(k_cache), _ptr(v_cache), code, _ptr(offsets), B, n_heads, 128,
                                      n_splits, _ptr(out), _ptr(lse), _stream(stream)))
    return out


def attention_noalloc_status(stream=None) -> int:
    """fsx_attention_noalloc_status: synchronises the stream, returns and clears the
    device status word of the static scratch (FSX_OK, FSX_ERR_DEVICE_ARG or FSX_ERR_TIMEOUT)."""
    return int(lib().fsx_attention_noalloc_status(_stream(stream)))


class Append:
    """Owns one fsx_append handle: the backbone's incremental cache append
    (weights uploaded at construction). Argument marshalling only."""

    def __init__(self, dims, weights: dict, max_batch: int, max_cache_rows: int, device: int = 0):
        self.dims = dims
        self.cfg = AppendConfig(dims.n_layers, dims.d_model, dims.n_heads, dims.head_dim, dims.d_ff, dims.n_new,
                                max_batch, max_cache_rows, float(dims.rope_base))
        keep = {k: np.ascontiguousarray(weights[k], dtype=np.float32) for k in _APPEND_WEIGHT_FIELDS}
        wst = AppendWeights(*[keep[k].ctypes.data_as(ctypes.POINTER(ctypes.c_float)) for k in _APPEND_WEIGHT_FIELDS])
        h = ctypes.c_void_p()
        check(lib().fsx_append_create(ctypes.byref(self.cfg), ctypes.byref(wst), device, ctypes.byref(h)))
        self.h = h
        del keep

    def close(self):
        if getattr(self, "h", None) and self.h.value:
            lib().fsx_append_destroy(self.h)
            self.h = ctypes.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def append(self, k_layers, v_layers, offsets, dst_rows, x_new, hidden, stream=None):
        B = int(x_new.shape[0])
        check(lib().fsx_append(self.h, _ptr_array(k_layers), _ptr_array(v_layers), _ptr(offsets), _ptr(dst_rows), B,
                               _ptr(x_new), _ptr(hidden), _stream(stream)))
        return hidden

    def status(self, stream=None) -> int:
        return lib().fsx_append_get_status(self.h, _stream(stream))

    def weight_bytes(self) -> int:
        return int(lib().fsx_append_weight_bytes(self.h))


class Session:
    """An fsx_session: the asynchronous fast-slow schedule of one vehicle over one cache
    (ticks on a snapshot of the committed rows, appends behind them). Marshalling only."""

    def __init__(self, expert: "Expert", append: "Append", k_layers, v_layers, capacity_rows: int,
                 committed_rows: int, concurrent: bool, device: int = 0):
        self._keep = (list(k_layers), list(v_layers))
        h = ctypes.c_void_p()
        check(lib().fsx_session_create(expert.h, append.h, _ptr_array(k_layers), _ptr_array(v_layers),
                                       len(k_layers), append.dims.n_new, capacity_rows, committed_rows,
                                       FSX_SCHED_CONCURRENT if concurrent else FSX_SCHED_SERIAL, device,
                                       ctypes.byref(h)))
        self.h = h

    def close(self):
        if getattr(self, "h", None) and self.h.value:
            lib().fsx_session_destroy(self.h)
            self.h = ctypes.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def append(self, x_new, hidden):
        check(lib().fsx_session_append(self.h, _ptr(x_new), _ptr(hidden)))

    def tick(self, frames, out) -> int:
        snap = ctypes.c_longlong()
        check(lib().fsx_session_tick(self.h, _ptr(frames), _ptr(out), ctypes.byref(snap)))
        return int(snap.value)

    def committed(self) -> int:
        return int(lib().fsx_session_committed(self.h))

    def reserved(self) -> int:
        return int(lib().fsx_session_reserved(self.h))

    def tick_stream(self) -> int:
        return lib().fsx_session_tick_stream(self.h)

    def append_stream(self) -> int:
        return lib().fsx_session_append_stream(self.h)

    def sync(self):
        check(lib().fsx_session_sync(self.h))
