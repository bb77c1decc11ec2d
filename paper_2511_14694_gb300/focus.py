"""Thin ctypes binding of libfocus.so (C ABI in include/focus.h).

Argument marshalling only: torch tensors are passed as raw device pointers and
the current torch stream as a cudaStream_t; every step of the compute path
runs in the library's CUDA kernels. There is no CPU fallback: if the library
cannot be loaded, every call raises.
"""
from __future__ import annotations

import ctypes
import math
import os

import numpy as np
import torch

from . import _build

FOCUS_OK = 0
STATUS_NAMES = {0: "ok", 1: "invalid argument", 2: "unsupported", 3: "capacity", 4: "cuda", 5: "timeout",
                6: "layout"}
LAYOUT_CLOSE_TAIL = 1
PREFILL_LEGACY_MMA = 1
PREFILL_KMER_LOCAL = 2
SUMMARY_TOKEN = 4


class FocusError(RuntimeError):
    def __init__(self, fn: str, code: int):
        super().__init__(f"{fn} failed: {STATUS_NAMES.get(code, code)} ({code})")
        self.code = code


_P = ctypes.c_void_p
_i32, _i64, _u32, _f32 = ctypes.c_int32, ctypes.c_int64, ctypes.c_uint32, ctypes.c_float


class LayoutOut(ctypes.Structure):
    _fields_ = [("T", _i64), ("R", _i64), ("kind", _P), ("src", _P), ("pos", _P), ("win", _P), ("tok", _P),
                ("keep", _P), ("win_off", _P), ("ring_off", _P), ("sum_idx", _P), ("base_off", _P)]


class CacheDesc(ctypes.Structure):
    _fields_ = [("ring_k", _P), ("ring_v", _P), ("win_k", _P), ("win_v", _P), ("ring_len", _P),
                ("win_fill", _P), ("win_idx", _P), ("k_per_window", _P), ("n_windows", _i32), ("W", _i32),
                ("B", _i32), ("H", _i32), ("d", _i32), ("C_ring", _i32), ("C_win", _i32), ("tail", _i32),
                ("pos_base", _P), ("rope_theta", _f32), ("W_per_window", _P), ("q_per_kv", _i32)]


class PrefillArgs(ctypes.Structure):
    _fields_ = [("q", _P), ("k", _P), ("v", _P), ("o", _P), ("lse", _P), ("T_span", _i64), ("d_win_off", _P),
                ("d_ring_off", _P), ("n_windows", _i32), ("w_begin", _i32), ("w_end", _i32), ("max_rows", _i32),
                ("scale", _f32), ("flags", _u32), ("workspace", _P), ("workspace_bytes", ctypes.c_size_t),
                ("h_k_per_window", _P)]


class PrefillHostArgs(ctypes.Structure):
    _fields_ = [("h_nt", _P), ("h_q", _P), ("h_k", _P), ("h_v", _P), ("h_o", _P), ("h_lse", _P),
                ("d_nt", _P), ("d_q", _P), ("d_k", _P), ("d_v", _P), ("d_o", _P), ("d_lse", _P),
                ("n_nt", _i64), ("W", _i32), ("d_W_sched", _P), ("n_windows", _i32), ("d_k_sched", _P),
                ("layout_flags", _u32), ("tail", _i32), ("layout", ctypes.POINTER(LayoutOut)), ("max_rows", _i32),
                ("scale", _f32), ("prefill_flags", _u32), ("workspace", _P), ("workspace_bytes", ctypes.c_size_t),
                ("groups", _i32), ("copy_in", _P), ("copy_out", _P)]


class CompactArgs(ctypes.Structure):
    _fields_ = [("src_k", _P), ("src_v", _P), ("src_T", _i64), ("src_row0", _i64), ("d_sum_idx", _P),
                ("d_ring_off", _P), ("n_windows", _i32), ("w_begin", _i32), ("w_end", _i32)]


_lib = None


def lib_path() -> str:
    return _build.LIB


def load() -> ctypes.CDLL:
    """Load libfocus.so (building it first if it is missing or stale)."""
    global _lib
    if _lib is not None:
        return _lib
    if _build.is_stale():
        _build.build()
    lib = ctypes.CDLL(_build.LIB)
    lib.focus_version.restype = _i32
    lib.focus_status_string.restype = ctypes.c_char_p
    lib.focus_status_string.argtypes = [ctypes.c_int]
    lib.focus_get_device_status.restype = ctypes.c_int
    lib.focus_get_device_status.argtypes = [_P, _i32, _P]
    lib.focus_layout_windows.restype = ctypes.c_int
    lib.focus_layout_windows.argtypes = [_i64, _i32, _P]
    lib.focus_layout_windows_sched.restype = ctypes.c_int
    lib.focus_layout_windows_sched.argtypes = [_i64, _i32, _P, _P]
    lib.focus_layout_size.restype = ctypes.c_int
    lib.focus_layout_size.argtypes = [_i64, _i32, _i32, _P, _u32, _i32, _P, _P, _P]
    lib.focus_layout.restype = ctypes.c_int
    lib.focus_layout.argtypes = [_i64, _i32, _i32, _P, _u32, _i32, _i32, _P, ctypes.POINTER(LayoutOut), _P]
    lib.focus_layout_size_sched.restype = ctypes.c_int
    lib.focus_layout_size_sched.argtypes = [_i64, _i32, _P, _P, _u32, _i32, _P, _P, _P]
    lib.focus_layout_sched.restype = ctypes.c_int
    lib.focus_layout_sched.argtypes = [_i64, _i32, _P, _P, _u32, _i32, _i32, _P, ctypes.POINTER(LayoutOut), _P]
    lib.focus_attn_prefill.restype = ctypes.c_int
    lib.focus_attn_prefill.argtypes = [ctypes.POINTER(CacheDesc), ctypes.POINTER(PrefillArgs), _P]
    lib.focus_prefill_kernel.restype = ctypes.c_int
    lib.focus_prefill_kernel.argtypes = [ctypes.POINTER(CacheDesc), ctypes.POINTER(PrefillArgs), _P]
    lib.focus_prefill_workspace_size.restype = ctypes.c_size_t
    lib.focus_prefill_workspace_size.argtypes = [ctypes.POINTER(CacheDesc), ctypes.POINTER(PrefillArgs)]
    lib.focus_prefill_host.restype = ctypes.c_int
    lib.focus_prefill_host.argtypes = [ctypes.POINTER(CacheDesc), ctypes.POINTER(PrefillHostArgs), _P]
    lib.focus_decode_workspace_size.restype = ctypes.c_size_t
    lib.focus_decode_workspace_size.argtypes = [ctypes.POINTER(CacheDesc)]
    lib.focus_attn_decode.restype = ctypes.c_int
    lib.focus_attn_decode.argtypes = [ctypes.POINTER(CacheDesc), _P, _P, _P, _f32, _P, _P, _P, ctypes.c_size_t, _P]
    lib.focus_attn_decode_noalloc.restype = ctypes.c_int
    lib.focus_attn_decode_noalloc.argtypes = [ctypes.POINTER(CacheDesc), _P, _P, _P, _f32, _P, _P, _P]
    lib.focus_kv_compact.restype = ctypes.c_int
    lib.focus_kv_compact.argtypes = [ctypes.POINTER(CacheDesc), ctypes.POINTER(CompactArgs), _P]
    lib.focus_selftest_timeout.restype = ctypes.c_int
    lib.focus_selftest_timeout.argtypes = [ctypes.c_uint64, _P]
    lib.focus_embed_tokens.restype = ctypes.c_int
    lib.focus_embed_tokens.argtypes = [_P, _i64, _P, _i32, _i32, _P, _P]
    _lib = lib
    return lib


def _check(fn: str, code: int):
    if code != FOCUS_OK:
        raise FocusError(fn, code)


def _ptr(t) -> int | None:
    if t is None:
        return None
    if isinstance(t, np.ndarray):
        return t.ctypes.data
    return t.data_ptr()


def _stream(stream=None) -> int:
    s = stream if stream is not None else torch.cuda.current_stream()
    return s.cuda_stream


def _cuda(t: torch.Tensor, name: str, dtype=None):
    if not (isinstance(t, torch.Tensor) and t.is_cuda and t.is_contiguous()):
        raise ValueError(f"{name} must be a contiguous CUDA tensor")
    if dtype is not None and t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    return t


# ----------------------------------------------------------------------------- layout

def n_windows(N: int, W) -> int:
    """M, the windows that cover N bases (focus_layout_windows, or
    focus_layout_windows_sched for a per-window sequence W)."""
    lib = load()
    M = _i32()
    if np.ndim(W) == 0:
        _check("focus_layout_windows", lib.focus_layout_windows(int(N), int(W), ctypes.byref(M)))
    else:
        Ws = np.ascontiguousarray(np.asarray(W, dtype=np.int32).reshape(-1))
        _check("focus_layout_windows_sched",
               lib.focus_layout_windows_sched(int(N), int(Ws.size), Ws.ctypes.data, ctypes.byref(M)))
    return M.value


def window_lengths(N: int, W):
    """None for windows of one integer length W; for a per-window sequence W
    (adaptive windowing) the int32 lengths of the windows that cover N bases (the
    library's count of them, focus_layout_windows_sched)."""
    if np.ndim(W) == 0:
        return None
    Ws = np.asarray(W, dtype=np.int32).reshape(-1)
    return np.ascontiguousarray(Ws[:n_windows(N, Ws)])


def layout_size(N: int, W, k_sched, close_tail: bool = True, tail: int = 0):
    """(T, R, M, max_rows) of the augmented layout (host arithmetic in the
    library). W: one window length, or a per-window sequence."""
    lib = load()
    Ws = window_lengths(N, W)
    M = n_windows(N, W) if Ws is None else int(Ws.size)
    k = np.ascontiguousarray(np.broadcast_to(np.asarray(k_sched, dtype=np.int32), (M,)))
    T, R, mx = _i64(), _i64(), _i32()
    flags = LAYOUT_CLOSE_TAIL if close_tail else 0
    if Ws is None:
        _check("focus_layout_size", lib.focus_layout_size(N, int(W), M, k.ctypes.data, flags, int(tail),
                                                          ctypes.byref(T), ctypes.byref(R), ctypes.byref(mx)))
    else:
        _check("focus_layout_size_sched", lib.focus_layout_size_sched(N, M, Ws.ctypes.data, k.ctypes.data, flags,
                                                                      int(tail), ctypes.byref(T), ctypes.byref(R),
                                                                      ctypes.byref(mx)))
    return T.value, R.value, M, mx.value


def layout_alloc(N: int, W, k_sched, B: int = 0, close_tail: bool = True, device="cuda", tail: int = 0) -> dict:
    """Allocate the device outputs of focus_layout (sizes from focus_layout_size)."""
    T, R, M, mx = layout_size(N, W, k_sched, close_tail, tail)
    Ws = window_lengths(N, W)
    k_host = np.ascontiguousarray(np.broadcast_to(np.asarray(k_sched, dtype=np.int32), (M,)))
    out = dict(
        kind=torch.empty(T, dtype=torch.uint8, device=device), keep=torch.empty(T, dtype=torch.uint8, device=device),
        src=torch.empty(T, dtype=torch.int32, device=device),
        pos=torch.empty(T, dtype=torch.int32, device=device), win=torch.empty(T, dtype=torch.int32, device=device),
        tok=torch.empty((B, T), dtype=torch.uint8, device=device) if B else None,
        win_off=torch.empty(M + 1, dtype=torch.int32, device=device),
        ring_off=torch.empty(M + 1, dtype=torch.int32, device=device),
        base_off=torch.empty(M + 1, dtype=torch.int32, device=device),
        W_dev=None if Ws is None else torch.from_numpy(Ws.copy()).to(device),
        sum_idx_buf=torch.empty(max(R, 1), dtype=torch.int32, device=device),
        k=torch.from_numpy(k_host.copy()).to(device))
    out["sum_idx"] = out["sum_idx_buf"][:R]
    out.update(T=T, R=R, M=M, max_rows=mx, k_host=k_host, N=N, W=W, W_host=Ws, B=B, close_tail=close_tail, tail=tail)
    return out


def _layout_desc(L: dict, with_tok: bool) -> LayoutOut:
    return LayoutOut(L["T"], L["R"], _ptr(L["kind"]), _ptr(L["src"]), _ptr(L["pos"]), _ptr(L["win"]),
                     _ptr(L["tok"]) if with_tok else None, _ptr(L["keep"]), _ptr(L["win_off"]),
                     _ptr(L["ring_off"]), _ptr(L["sum_idx_buf"]), _ptr(L["base_off"]))


def layout_run(L: dict, nt: torch.Tensor | None = None, stream=None) -> None:
    """Launch focus_layout into buffers from layout_alloc (asynchronous)."""
    lib = load()
    if nt is not None:
        _cuda(nt, "nt", torch.uint8)
        if L["tok"] is None or tuple(nt.shape) != (L["B"], L["N"]):
            raise ValueError("nt shape does not match the allocated layout")
    desc = _layout_desc(L, nt is not None)
    flags = LAYOUT_CLOSE_TAIL if L["close_tail"] else 0
    B = 0 if nt is None else L["B"]
    if L["W_dev"] is None:
        _check("focus_layout", lib.focus_layout(L["N"], int(L["W"]), L["M"], _ptr(L["k"]), flags, int(L["tail"]), B,
                                                _ptr(nt), ctypes.byref(desc), _stream(stream)))
    else:
        _check("focus_layout_sched", lib.focus_layout_sched(L["N"], L["M"], _ptr(L["W_dev"]), _ptr(L["k"]), flags,
                                                            int(L["tail"]), B, _ptr(nt), ctypes.byref(desc),
                                                            _stream(stream)))


def layout(N: int, W: int, k_sched, nt: torch.Tensor | None = None, close_tail: bool = True,
           device="cuda", stream=None, tail: int = 0) -> dict:
    """Build the augmented token layout on the device (focus_layout) and keep host
    copies of the window/ring offsets for slicing per-window inputs (syncs)."""
    L = layout_alloc(N, W, k_sched, 0 if nt is None else int(nt.shape[0]), close_tail, device, tail)
    layout_run(L, nt, stream)
    L["win_off_host"] = L["win_off"].cpu().numpy()
    L["ring_off_host"] = L["ring_off"].cpu().numpy()
    L["base_off_host"] = L["base_off"].cpu().numpy()
    return L


# ----------------------------------------------------------------------------- cache

class Cache:
    """Caller-owned compressed KV cache (ring of retained FOCUS K/V + the
    current window buffer) and its C descriptor."""

    def __init__(self, B: int, H: int, d: int, C_ring: int, C_win: int = 0, W: int = 0, k_sched=None,
                 device="cuda", tail: int = 0, rope_theta: float = 0.0, W_sched=None, q_per_kv: int = 1):
        """``rope_theta`` > 0 turns on the rotary embedding of queries and keys at
        their position ids; ``pos_base`` [B] (zeros here) holds the position id of
        each sequence's current decode window's first row. ``W_sched`` (one length
        per window, adaptive windowing) replaces the fixed W for decode and
        window-mode compaction. ``q_per_kv`` query heads share each of the H K/V
        heads (grouped-query heads): queries and outputs have H * q_per_kv heads."""
        self.q_per_kv = int(q_per_kv)
        self.B, self.H, self.d, self.C_ring, self.C_win, self.W, self.tail = B, H, d, C_ring, C_win, W, tail
        self.rope_theta = float(rope_theta)
        bf = dict(dtype=torch.bfloat16, device=device)
        self.ring_k = torch.zeros((B, H, max(C_ring, 1), d), **bf)
        self.ring_v = torch.zeros((B, H, max(C_ring, 1), d), **bf)
        self.win_k = torch.zeros((B, H, max(C_win, 1), d), **bf) if C_win else None
        self.win_v = torch.zeros((B, H, max(C_win, 1), d), **bf) if C_win else None
        self.ring_len = torch.zeros(B, dtype=torch.int32, device=device)
        self.win_fill = torch.zeros(B, dtype=torch.int32, device=device)
        self.win_idx = torch.zeros(B, dtype=torch.int32, device=device)
        self.pos_base = torch.zeros(B, dtype=torch.int32, device=device)
        self.W_sched = (None if W_sched is None else
                        torch.from_numpy(np.asarray(W_sched, dtype=np.int32).reshape(-1).copy()).to(device))
        ks = np.zeros(1, np.int32) if k_sched is None else np.asarray(k_sched, dtype=np.int32).reshape(-1)
        self.k_sched = torch.from_numpy(ks.copy()).to(device)
        self.desc = CacheDesc(_ptr(self.ring_k), _ptr(self.ring_v), _ptr(self.win_k), _ptr(self.win_v),
                              _ptr(self.ring_len), _ptr(self.win_fill), _ptr(self.win_idx), _ptr(self.k_sched),
                              int(self.k_sched.numel()), W, B, H, d, C_ring, C_win, tail, _ptr(self.pos_base),
                              self.rope_theta, _ptr(self.W_sched), self.q_per_kv)

    _STATE = ("ring_k", "ring_v", "win_k", "win_v", "ring_len", "win_fill", "win_idx", "pos_base")

    def snapshot(self) -> dict:
        """Copies of the cache state (ring and window K/V, ring_len, win_fill,
        win_idx, pos_base) on the same device: a checkpoint of a decode stream."""
        return {n: getattr(self, n).clone() for n in self._STATE if getattr(self, n) is not None}

    def restore(self, state: dict) -> None:
        """Copy a snapshot back in place (same shapes); decoding then continues
        exactly as from the moment the snapshot was taken."""
        for n, t in state.items():
            getattr(self, n).copy_(t)

    def part(self, b0: int = 0, b1: int | None = None, h0: int = 0, h1: int | None = None) -> "Cache":
        """A view of sequences [b0, b1) and K/V heads [h0, h1) sharing this cache's
        memory, for calls that process the cache in groups. The part must be
        contiguous in the [B, H, rows, d] buffers: all heads, or one sequence."""
        b1 = self.B if b1 is None else b1
        h1 = self.H if h1 is None else h1
        if not (0 <= b0 < b1 <= self.B and 0 <= h0 < h1 <= self.H):
            raise ValueError(f"cache part [{b0}, {b1}) x [{h0}, {h1}) outside B={self.B}, H={self.H}")
        if (h0, h1) != (0, self.H) and b1 - b0 != 1:
            raise ValueError("a head range needs a single sequence (the part must be contiguous)")
        v = object.__new__(Cache)
        v.__dict__.update(self.__dict__)
        v.B, v.H = b1 - b0, h1 - h0
        for name in ("ring_k", "ring_v", "win_k", "win_v"):
            t = getattr(self, name)
            setattr(v, name, None if t is None else t[b0:b1, h0:h1])
        for name in ("ring_len", "win_fill", "win_idx", "pos_base"):
            setattr(v, name, getattr(self, name)[b0:b1])
        v.desc = CacheDesc(_ptr(v.ring_k), _ptr(v.ring_v), _ptr(v.win_k), _ptr(v.win_v), _ptr(v.ring_len),
                           _ptr(v.win_fill), _ptr(v.win_idx), _ptr(self.k_sched), int(self.k_sched.numel()), self.W,
                           v.B, v.H, self.d, self.C_ring, self.C_win, self.tail, _ptr(v.pos_base), self.rope_theta,
                           _ptr(self.W_sched), self.q_per_kv)
        return v

    def workspace_bytes(self) -> int:
        return int(load().focus_decode_workspace_size(ctypes.byref(self.desc)))

    def new_workspace(self) -> torch.Tensor:
        n = self.workspace_bytes()
        return torch.empty(max(n, 16) // 4 + 4, dtype=torch.float32, device=self.ring_k.device)


# ----------------------------------------------------------------------------- verbs

def _check_heads(cache: Cache, q, k, v):
    g = max(cache.q_per_kv, 1)
    if q.shape[1] != cache.H * g or k.shape[1] != cache.H or v.shape[1] != cache.H:
        raise ValueError(f"heads: q {q.shape[1]} (want {cache.H * g}), k {k.shape[1]}, v {v.shape[1]} "
                         f"(want {cache.H})")


def _prefill_args(q, k, v, o, lse, L: dict, w_begin: int, w_end: int, scale: float, flags: int, workspace=None,
                  host_schedule: bool = True):
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    # the host copy of the cadence schedule lets the k-mer-local mode pick its k-mer-tiled kernel
    return PrefillArgs(_ptr(q), _ptr(k), _ptr(v), _ptr(o), _ptr(lse), q.shape[2], _ptr(L["win_off"]),
                       _ptr(L["ring_off"]), L["M"], w_begin, w_end, int(L["max_rows"]), scale, flags,
                       _ptr(workspace), ws_bytes, _ptr(L["k_host"]) if host_schedule else None)


def prefill_workspace_bytes(cache: Cache, q, k, v, L: dict, w_begin: int = 0, w_end: int | None = None,
                            flags: int = 0, host_schedule: bool = True) -> int:
    """focus_prefill_workspace_size: device workspace bytes that let these
    arguments use the fastest kernel (0: none needed)."""
    w_end = L["M"] if w_end is None else w_end
    a = _prefill_args(q, k, v, q, None, L, w_begin, w_end, 1.0 / math.sqrt(q.shape[3]), flags,
                      host_schedule=host_schedule)
    return int(load().focus_prefill_workspace_size(ctypes.byref(cache.desc), ctypes.byref(a)))


def new_prefill_workspace(cache: Cache, q, k, v, L: dict, w_begin: int = 0, w_end: int | None = None,
                          flags: int = 0, host_schedule: bool = True):
    """A device buffer of prefill_workspace_bytes (None when none is needed)."""
    n = prefill_workspace_bytes(cache, q, k, v, L, w_begin, w_end, flags, host_schedule)
    return None if n == 0 else torch.empty(n, dtype=torch.uint8, device=q.device)


def attn_prefill(cache: Cache, q, k, v, L: dict, w_begin: int = 0, w_end: int | None = None, scale=None,
                 o=None, lse=None, flags: int = 0, stream=None, workspace="auto", host_schedule: bool = True):
    """focus_attn_prefill over windows [w_begin, w_end). q/k/v: bf16 [B, H, T_span, d]
    holding the augmented rows of those windows. Returns (o, lse).
    ``workspace``: a device buffer for the library (see prefill_workspace_bytes),
    None for none, or "auto" to allocate one when the arguments can use it.
    ``host_schedule``: pass the layout's host copy of the k schedule
    (h_k_per_window), which the k-mer-local mode's k-mer-tiled kernel needs."""
    lib = load()
    w_end = L["M"] if w_end is None else w_end
    for name, t in (("q", q), ("k", k), ("v", v)):
        _cuda(t, name, torch.bfloat16)
    _check_heads(cache, q, k, v)
    B, H, T_span, d = q.shape
    if o is None:
        o = torch.empty_like(q)
    if lse is None:
        lse = torch.empty((B, H, T_span), dtype=torch.float32, device=q.device)
    scale = 1.0 / math.sqrt(d) if scale is None else float(scale)
    if isinstance(workspace, str):
        workspace = new_prefill_workspace(cache, q, k, v, L, w_begin, w_end, flags, host_schedule)
        if workspace is not None and stream is not None:
            # allocated on the current stream, used on `stream`: keep the caching
            # allocator from reusing it before the launch there is done
            workspace.record_stream(stream)
    elif workspace is not None:
        _cuda(workspace, "workspace")
    a = _prefill_args(q, k, v, o, lse, L, w_begin, w_end, scale, flags, workspace, host_schedule)
    _check("focus_attn_prefill", lib.focus_attn_prefill(ctypes.byref(cache.desc), ctypes.byref(a), _stream(stream)))
    return o, lse


def prefill_host(cache: Cache, L: dict, host: dict, dev: dict, copy_in, copy_out, groups: int = 8, scale=None,
                 flags: int = 0, workspace="auto", stream=None):
    """focus_prefill_host: the masked-parallel prefill of a layer whose inputs and
    outputs are in (pinned) host memory. host["nt"] (uint8 [B, N]),
    host["q"/"k"/"v"] (bf16 [B, H, T, d]) in; host["o"] (bf16) and host["lse"]
    (fp32 [B, H, T], or None) out; ``dev`` holds device tensors of the same
    shapes; L from layout_alloc (its tok is written). The library copies each
    group of heads (B = 1) or sequences in on ``copy_in``, runs its compaction and
    attention on ``stream`` and copies it out on ``copy_out``; work is only
    enqueued, and once ``stream`` is done, so is everything."""
    lib = load()
    for name in ("nt", "q", "k", "v", "o"):
        if not (isinstance(host[name], torch.Tensor) and not host[name].is_cuda and host[name].is_contiguous()):
            raise ValueError(f"host[{name!r}] must be a contiguous host tensor")
        _cuda(dev[name], f"dev[{name!r}]")
        if tuple(host[name].shape) != tuple(dev[name].shape):
            raise ValueError(f"host[{name!r}] and dev[{name!r}] differ in shape")
    _check_heads(cache, dev["q"], dev["k"], dev["v"])
    if tuple(dev["nt"].shape) != (L["B"], L["N"]) or L["tok"] is None:
        raise ValueError("nt shape does not match the allocated layout")
    d = dev["q"].shape[-1]
    scale = 1.0 / math.sqrt(d) if scale is None else float(scale)
    if isinstance(workspace, str):
        workspace = new_prefill_workspace(cache, dev["q"], dev["k"], dev["v"], L, flags=flags)
        if workspace is not None and stream is not None:
            workspace.record_stream(stream)          # used on `stream`, allocated on the current one
    desc = _layout_desc(L, True)
    lse_h, lse_d = host.get("lse"), dev.get("lse")
    a = PrefillHostArgs(_ptr(host["nt"]), _ptr(host["q"]), _ptr(host["k"]), _ptr(host["v"]), _ptr(host["o"]),
                        _ptr(lse_h), _ptr(dev["nt"]), _ptr(dev["q"]), _ptr(dev["k"]), _ptr(dev["v"]),
                        _ptr(dev["o"]), _ptr(lse_d) if lse_h is not None else None, L["N"],
                        0 if L["W_dev"] is not None else int(L["W"]), _ptr(L["W_dev"]), L["M"], _ptr(L["k"]),
                        LAYOUT_CLOSE_TAIL if L["close_tail"] else 0, int(L["tail"]), ctypes.pointer(desc),
                        int(L["max_rows"]), scale, flags, _ptr(workspace),
                        0 if workspace is None else workspace.numel() * workspace.element_size(), int(groups),
                        copy_in.cuda_stream, copy_out.cuda_stream)
    _check("focus_prefill_host", lib.focus_prefill_host(ctypes.byref(cache.desc), ctypes.byref(a), _stream(stream)))
    return host["o"], lse_h


PREFILL_KERNELS = {0: "legacy mma.sync", 1: "tcgen05, one CTA per work item", 2: "tcgen05 persistent",
                   3: "tcgen05 k-mer tiles"}
PREFILL_KERNEL_ROTATION_PASS = 16


def prefill_kernel(cache: Cache, q, k, v, L: dict, w_begin: int = 0, w_end: int | None = None, flags: int = 0,
                   o=None, workspace="auto", host_schedule: bool = True) -> str:
    """Name of the kernel focus_attn_prefill would launch for these arguments
    (focus_prefill_kernel: host only, nothing runs on the device), prefixed with
    "rotation pass + " when a rotary-embedding pass runs before it. ``workspace``
    as for attn_prefill; "auto" assumes the workspace attn_prefill would allocate."""
    lib = load()
    w_end = L["M"] if w_end is None else w_end
    a = _prefill_args(q, k, v, q if o is None else o, None, L, w_begin, w_end, 1.0 / math.sqrt(q.shape[3]), flags,
                      host_schedule=host_schedule)
    if isinstance(workspace, str):
        a.workspace_bytes = prefill_workspace_bytes(cache, q, k, v, L, w_begin, w_end, flags, host_schedule)
        a.workspace = 16 if a.workspace_bytes else None        # a placeholder address: nothing is launched
    elif workspace is not None:
        a.workspace, a.workspace_bytes = _ptr(workspace), workspace.numel() * workspace.element_size()
    out = ctypes.c_int32()
    _check("focus_prefill_kernel", lib.focus_prefill_kernel(ctypes.byref(cache.desc), ctypes.byref(a),
                                                           ctypes.byref(out)))
    name = PREFILL_KERNELS[out.value & ~PREFILL_KERNEL_ROTATION_PASS]
    return "rotation pass + " + name if out.value & PREFILL_KERNEL_ROTATION_PASS else name


def embed_tokens(tok, table, out=None, stream=None):
    """focus_embed_tokens: out[..., :] = table[tok[...]] for the layout's token
    stream (uint8, any shape, e.g. L["tok"] [B, T]) and a bf16 table
    [n_tokens, D]; returns out (bf16 [*tok.shape, D])."""
    lib = load()
    _cuda(tok, "tok", torch.uint8)
    _cuda(table, "table", torch.bfloat16)
    n_tokens, D = table.shape
    if out is None:
        out = torch.empty((*tok.shape, D), dtype=torch.bfloat16, device=tok.device)
    _cuda(out, "out", torch.bfloat16)
    if tuple(out.shape) != (*tok.shape, D):
        raise ValueError(f"out shape {tuple(out.shape)}, want {(*tok.shape, D)}")
    _check("focus_embed_tokens", lib.focus_embed_tokens(_ptr(tok), tok.numel(), _ptr(table), n_tokens, D, _ptr(out),
                                                        _stream(stream)))
    return out


def kv_compact_bulk(cache: Cache, src_k, src_v, L: dict, w_begin: int = 0, w_end: int | None = None,
                    src_row0: int = 0, stream=None):
    """focus_kv_compact, bulk mode: gather the FOCUS rows of windows
    [w_begin, w_end) of src into the ring."""
    lib = load()
    w_end = L["M"] if w_end is None else w_end
    _cuda(src_k, "src_k", torch.bfloat16)
    _cuda(src_v, "src_v", torch.bfloat16)
    a = CompactArgs(_ptr(src_k), _ptr(src_v), int(src_k.shape[2]), int(src_row0), _ptr(L["sum_idx_buf"]),
                    _ptr(L["ring_off"]), L["M"], w_begin, w_end)
    _check("focus_kv_compact", lib.focus_kv_compact(ctypes.byref(cache.desc), ctypes.byref(a), _stream(stream)))


def kv_compact_window(cache: Cache, stream=None):
    """focus_kv_compact, window mode: retire every full window buffer."""
    lib = load()
    a = CompactArgs(None, None, 0, 0, None, None, 0, 0, 0)
    _check("focus_kv_compact", lib.focus_kv_compact(ctypes.byref(cache.desc), ctypes.byref(a), _stream(stream)))


def attn_decode(cache: Cache, q, k_new, v_new, scale=None, o=None, lse=None, workspace=None, stream=None):
    """focus_attn_decode: one new token per sequence. q/k_new/v_new: bf16 [B, H, d]."""
    lib = load()
    for name, t in (("q", q), ("k_new", k_new), ("v_new", v_new)):
        _cuda(t, name, torch.bfloat16)
    _check_heads(cache, q, k_new, v_new)
    if o is None:
        o = torch.empty_like(q)
    if lse is None:
        lse = torch.empty(q.shape[:2], dtype=torch.float32, device=q.device)
    if workspace is None:
        workspace = cache.new_workspace()
    scale = 1.0 / math.sqrt(q.shape[-1]) if scale is None else float(scale)
    _check("focus_attn_decode",
           lib.focus_attn_decode(ctypes.byref(cache.desc), _ptr(q), _ptr(k_new), _ptr(v_new), scale, _ptr(o),
                                 _ptr(lse), _ptr(workspace), workspace.numel() * workspace.element_size(),
                                 _stream(stream)))
    return o, lse


def attn_decode_noalloc(cache: Cache, q, k_new, v_new, scale=None, o=None, lse=None, stream=None):
    """focus_attn_decode_noalloc: same as attn_decode, but the library keeps the
    split-K scratch in its own fixed device array, so the caller passes no
    workspace (for callers that cannot allocate device memory)."""
    lib = load()
    for name, t in (("q", q), ("k_new", k_new), ("v_new", v_new)):
        _cuda(t, name, torch.bfloat16)
    _check_heads(cache, q, k_new, v_new)
    if o is None:
        o = torch.empty_like(q)
    if lse is None:
        lse = torch.empty(q.shape[:2], dtype=torch.float32, device=q.device)
    scale = 1.0 / math.sqrt(q.shape[-1]) if scale is None else float(scale)
    _check("focus_attn_decode_noalloc",
           lib.focus_attn_decode_noalloc(ctypes.byref(cache.desc), _ptr(q), _ptr(k_new), _ptr(v_new), scale,
                                         _ptr(o), _ptr(lse), _stream(stream)))
    return o, lse


def selftest_timeout(limit_ns: int = 20_000_000, stream=None) -> None:
    """focus_selftest_timeout: a bounded device wait that nothing completes gives up
    after limit_ns and sets FOCUS_ERR_TIMEOUT in the device status word."""
    _check("focus_selftest_timeout", load().focus_selftest_timeout(int(limit_ns), _stream(stream)))


def device_status(clear: bool = True, stream=None) -> int:
    """Read (and by default clear) the sticky device status word; syncs the stream."""
    lib = load()
    v = _i32()
    _check("focus_get_device_status", lib.focus_get_device_status(ctypes.byref(v), int(clear), _stream(stream)))
    return v.value
