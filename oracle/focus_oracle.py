"""Python wrapper of the fp64 FOCUS oracle (``focus_oracle.c``).

TEST INFRASTRUCTURE ONLY: the test suite, ``__graft_entry__.smoke()`` and the
benchmark's ``cpu_baseline`` / ``--impl reference`` legs are its only users.
The product path (``paper_2511_14694_gb300``) never imports it.

Each function states the passage of arXiv 2511.14694 it follows; the C file
holds the arithmetic. Inputs are numpy arrays or CPU torch tensors; bf16
tensors are passed as their raw 16-bit patterns so the oracle widens exactly
the values the GPU read.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "focus_oracle.c")
_LIB_PATH = os.path.join(_HERE, "libfocus_oracle.so")
_lib = None

SUMMARY_TOKEN = 4


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (fp64, IEEE semantics, OpenMP over rows)."""
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fopenmp", "-fPIC", "-shared",
           "-fno-fast-math", _SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load(path: str | None = None):
    global _lib
    if _lib is not None and path is None:
        return _lib
    if path is None:
        build()
    lib = ctypes.CDLL(path or _LIB_PATH)
    P = ctypes.c_void_p
    i64, i32, f64 = ctypes.c_int64, ctypes.c_int32, ctypes.c_double
    lib.fo_layout_size.restype = i64
    lib.fo_layout_size.argtypes = [i64, i32, i32, P, i32, i32, P]
    lib.fo_layout.restype = i64
    lib.fo_layout.argtypes = [i64, i32, i32, P, i32, i32, i32, P, P, P, P, P, P, P, P, P, P]
    lib.fo_attn_rows.restype = None
    lib.fo_attn_rows.argtypes = [i64, i32, P, P, P, P, P, f64, i64, P, P, P, P]
    lib.fo_prefill_sequential.restype = i32
    lib.fo_prefill_sequential.argtypes = [i32, i32, P, P, P, P, P, f64, P, P, P, P, P, i64, P]
    lib.fo_decode.restype = None
    lib.fo_decode.argtypes = [i32, i64, P, P, i64, P, P, P, i64, P, P, P, P, f64, P, P]
    lib.fo_layout_size_sched.restype = i64
    lib.fo_layout_size_sched.argtypes = [i64, i32, P, P, i32, i32, P]
    lib.fo_layout_sched.restype = i64
    lib.fo_layout_sched.argtypes = [i64, i32, P, P, i32, i32, i32, P, P, P, P, P, P, P, P, P, P, P]
    lib.fo_layout_kmer_sched.restype = i64
    lib.fo_layout_kmer_sched.argtypes = [i64, i32, P, P, i32, P]
    lib.fo_layout_kmer.restype = i64
    lib.fo_layout_kmer.argtypes = [i64, i32, i32, P, i32, P]
    lib.fo_attn_rows_kmer_local.restype = None
    lib.fo_attn_rows_kmer_local.argtypes = [i64, i32, P, P, P, P, P, P, f64, i64, P, P, P, P]
    lib.fo_rope.restype = None
    lib.fo_rope.argtypes = [i64, i32, P, f64, i32, P, P]
    lib.fo_round_bf16.restype = f64
    lib.fo_round_bf16.argtypes = [f64]
    lib.fo_attn_rows_f64.restype = None
    lib.fo_attn_rows_f64.argtypes = [i64, i32, P, P, P, P, P, f64, i64, P, P, P, P]
    lib.fo_decode_f64.restype = None
    lib.fo_decode_f64.argtypes = [i32, i64, P, P, i64, P, P, P, i64, P, P, P, P, f64, P, P]
    lib.fo_window_retained_rows.restype = i32
    lib.fo_window_retained_rows.argtypes = [i64, i32, i32, i32, P, i32]
    _lib = lib
    return lib


class use_library:
    """Context manager: route every wrapper call to another build of the oracle
    (the mutation tests use it to check that the pins catch planted mistakes)."""

    def __init__(self, path: str):
        self.path = path

    def __enter__(self):
        global _lib
        self._saved = _lib
        _load(self.path)
        return self

    def __exit__(self, *exc):
        global _lib
        _lib = self._saved
        return False


def _ptr(a: np.ndarray | None):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _bits(x) -> np.ndarray:
    """bf16 tensor / uint16 array -> contiguous uint16 numpy array of raw bits."""
    if isinstance(x, np.ndarray):
        assert x.dtype == np.uint16, x.dtype
        return np.ascontiguousarray(x)
    import torch
    assert x.dtype == torch.bfloat16, x.dtype
    return np.ascontiguousarray(x.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16))


def _k_array(M: int, k_sched) -> np.ndarray:
    k = np.ascontiguousarray(np.broadcast_to(np.asarray(k_sched, dtype=np.int32), (M,)))
    return k


def n_windows(N: int, W: int) -> int:
    """M = ceil(L/W) (App. A)."""
    return (N + W - 1) // W


def window_schedule(N: int, W) -> np.ndarray:
    """Base lengths of the windows that cover N bases: M = ceil(N/W) copies of
    an integer W, or the shortest prefix of a per-window sequence W (adaptive
    windowing) whose sum reaches N."""
    if np.ndim(W) == 0:
        return np.full(n_windows(N, int(W)), int(W), np.int32)
    Ws = np.asarray(W, dtype=np.int64).reshape(-1)
    if N == 0:
        return np.zeros(0, np.int32)
    cover = np.cumsum(Ws)
    if cover.size == 0 or cover[-1] < N:
        raise ValueError("window schedule does not cover the sequence")
    M = int(np.searchsorted(cover, N) + 1)
    return np.ascontiguousarray(Ws[:M].astype(np.int32))


def layout_size(N: int, W, k_sched, close_tail: bool = True, tail: int = 0):
    """(T, R, M): augmented length, retained rows (summaries + boundary tails),
    windows (App. A). W: one window length, or a per-window schedule."""
    lib = _load()
    Ws = window_schedule(N, W)
    M = Ws.size
    k = _k_array(M, k_sched)
    R = np.zeros(1, np.int64)
    T = lib.fo_layout_size_sched(N, M, _ptr(Ws), _ptr(k), int(close_tail), int(tail), _ptr(R))
    if T < 0:
        raise ValueError("bad layout arguments")
    return int(T), int(R[0]), M


def layout(N: int, W, k_sched, nt=None, close_tail: bool = True, tail: int = 0) -> dict:
    """Token layout: summary insertion after every k bases per window (Sec. 3.2
    "Setup and tokens"; App. A). W: one window length or a per-window schedule.
    ``nt``: uint8 [B, N] nucleotide ids or None. ``tail``: ordinary rows kept at
    the end of each window (boundary tail)."""
    lib = _load()
    T, R, M = layout_size(N, W, k_sched, close_tail, tail)
    Ws = window_schedule(N, W)
    k = _k_array(M, k_sched)
    if nt is not None:
        nt = np.ascontiguousarray(np.asarray(nt, dtype=np.uint8).reshape(-1, N))
        B = nt.shape[0]
        tok = np.zeros((B, T), np.uint8)
    else:
        B, tok = 0, None
    out = dict(
        kind=np.zeros(T, np.uint8), keep=np.zeros(T, np.uint8), src=np.zeros(T, np.int32), pos=np.zeros(T, np.int32),
        win=np.zeros(T, np.int32), win_off=np.zeros(M + 1, np.int32),
        ring_off=np.zeros(M + 1, np.int32), sum_idx=np.zeros(max(R, 1), np.int32),
        base_off=np.zeros(M + 1, np.int32))
    t = lib.fo_layout_sched(N, M, _ptr(Ws), _ptr(k), int(close_tail), int(tail), B, _ptr(nt), _ptr(out["kind"]),
                            _ptr(out["src"]), _ptr(out["pos"]), _ptr(out["win"]), _ptr(tok), _ptr(out["keep"]),
                            _ptr(out["win_off"]), _ptr(out["ring_off"]), _ptr(out["sum_idx"]), _ptr(out["base_off"]))
    assert t == T
    out["sum_idx"] = out["sum_idx"][:R]
    out["tok"] = tok
    out.update(T=T, R=R, M=M, W_sched=Ws)
    return out


def attn_rows(q, k, v, keep, win, scale: float, heads, rows):
    """Masked-parallel attention at selected rows (App. A.1 (ii); Eq.
    focus-attn's visible set). q/k/v: bf16 [n_heads, T, d]; ``keep``: the layout's
    retained-row flags (FOCUS rows, plus boundary-tail rows if any).
    ``heads``/``rows``: equal-length integer sequences. Returns (o [n, d] fp64,
    lse [n] fp64)."""
    lib = _load()
    qb, kb, vb = _bits(q), _bits(k), _bits(v)
    nh, T, d = qb.shape
    keep = np.ascontiguousarray(keep, dtype=np.uint8)
    win = np.ascontiguousarray(win, dtype=np.int32)
    assert keep.shape == (T,) and win.shape == (T,)
    heads = np.ascontiguousarray(heads, dtype=np.int64)
    rows = np.ascontiguousarray(rows, dtype=np.int64)
    assert heads.shape == rows.shape
    assert heads.size == 0 or (heads.min() >= 0 and heads.max() < nh and rows.min() >= 0 and rows.max() < T)
    n = rows.size
    o = np.zeros((n, d), np.float64)
    lse = np.zeros(n, np.float64)
    lib.fo_attn_rows(T, d, _ptr(keep), _ptr(win), _ptr(qb), _ptr(kb), _ptr(vb), float(scale),
                     n, _ptr(heads), _ptr(rows), _ptr(o), _ptr(lse))
    return o, lse


def layout_kmer(N: int, W, k_sched, close_tail: bool = True) -> np.ndarray:
    """In-window k-mer index of every augmented row (Sec. 3.2 "Setup and
    tokens"): a base's own k-mer, the summarised k-mer for a FOCUS row; 0 for
    every row of a window with k = 0."""
    lib = _load()
    T, _, M = layout_size(N, W, k_sched, close_tail)
    Ws = window_schedule(N, W)
    k = _k_array(M, k_sched)
    out = np.zeros(max(T, 1), np.int32)
    t = lib.fo_layout_kmer_sched(N, M, _ptr(Ws), _ptr(k), int(close_tail), _ptr(out))
    if t < 0:
        raise ValueError("bad layout arguments")
    return out[:T]


def attn_rows_kmer_local(q, k, v, kind, win, kmer, scale: float, heads, rows):
    """Attention at selected rows under the main text's k-mer-local visibility
    (Sec. 3.2 "Visibility and summarization rule"): own k-mer (causal), the
    window's FOCUS rows, and the carried boundary (last FOCUS row of the previous
    window). Arguments and outputs as in ``attn_rows``; ``kind``/``win``/``kmer``
    are the layout's per-row arrays."""
    lib = _load()
    qb, kb, vb = _bits(q), _bits(k), _bits(v)
    nh, T, d = qb.shape
    kind = np.ascontiguousarray(kind, dtype=np.uint8)
    win = np.ascontiguousarray(win, dtype=np.int32)
    kmer = np.ascontiguousarray(kmer, dtype=np.int32)
    assert kind.shape == (T,) and win.shape == (T,) and kmer.shape == (T,)
    heads = np.ascontiguousarray(heads, dtype=np.int64)
    rows = np.ascontiguousarray(rows, dtype=np.int64)
    assert heads.shape == rows.shape
    assert heads.size == 0 or (heads.min() >= 0 and heads.max() < nh and rows.min() >= 0 and rows.max() < T)
    n = rows.size
    o = np.zeros((n, d), np.float64)
    lse = np.zeros(n, np.float64)
    lib.fo_attn_rows_kmer_local(T, d, _ptr(kind), _ptr(win), _ptr(kmer), _ptr(qb), _ptr(kb), _ptr(vb),
                                float(scale), n, _ptr(heads), _ptr(rows), _ptr(o), _ptr(lse))
    return o, lse


def prefill_sequential(q, k, v, win_off, keep, scale: float, want=None, ring_cap=None):
    """Sequential windowed form with KV retention (App. A.1 (i), App. A.2) for
    ONE head: q/k/v bf16 [T, d]; ``keep``: retained-row flags. Returns (o [T,d]
    fp64, lse [T] fp64, ring_k uint16 [R,d], ring_v uint16 [R,d]). Rows of
    windows not in ``want`` are NaN."""
    lib = _load()
    qb, kb, vb = _bits(q), _bits(k), _bits(v)
    T, d = qb.shape
    win_off = np.ascontiguousarray(win_off, dtype=np.int32)
    M = win_off.size - 1
    keep = np.ascontiguousarray(keep, dtype=np.uint8)
    cap = int(ring_cap if ring_cap is not None else max(int((keep == 1).sum()), 1))
    want_a = None if want is None else np.ascontiguousarray(want, dtype=np.uint8)
    o = np.full((T, d), np.nan)
    lse = np.full(T, np.nan)
    rk = np.zeros((cap, d), np.uint16)
    rv = np.zeros((cap, d), np.uint16)
    R = np.zeros(1, np.int64)
    rc = lib.fo_prefill_sequential(d, M, _ptr(win_off), _ptr(keep), _ptr(qb), _ptr(kb), _ptr(vb),
                                   float(scale), _ptr(want_a), _ptr(o), _ptr(lse), _ptr(rk), _ptr(rv),
                                   cap, _ptr(R))
    if rc != 0:
        raise ValueError("ring capacity too small")
    r = int(R[0])
    return o, lse, rk[:r], rv[:r]


def decode(q, k_new, v_new, ring_k, ring_v, R, win_k, win_v, fill, scale: float):
    """One decode step for n independent streams (App. A.2): the new row is
    appended after ``fill`` window rows and attends to ring[:R] ∪ window[:fill]
    ∪ itself. q/k_new/v_new: bf16 [n, d]; ring_*: bf16 [n, C_ring, d];
    win_*: bf16 [n, C_win, d]; R, fill: int [n]. Returns (o [n,d], lse [n])."""
    lib = _load()
    qb, knb, vnb = _bits(q), _bits(k_new), _bits(v_new)
    rkb, rvb, wkb, wvb = _bits(ring_k), _bits(ring_v), _bits(win_k), _bits(win_v)
    n, d = qb.shape
    R = np.ascontiguousarray(R, dtype=np.int64)
    fill = np.ascontiguousarray(fill, dtype=np.int64)
    assert R.shape == (n,) and fill.shape == (n,)
    assert (R <= rkb.shape[1]).all() and (fill < wkb.shape[1] + 1).all()
    o = np.zeros((n, d), np.float64)
    lse = np.zeros(n, np.float64)
    lib.fo_decode(d, n, _ptr(rkb), _ptr(rvb), rkb.shape[1], _ptr(R), _ptr(wkb), _ptr(wvb),
                  wkb.shape[1], _ptr(fill), _ptr(qb), _ptr(knb), _ptr(vnb), float(scale),
                  _ptr(o), _ptr(lse))
    return o, lse


def round_bf16(x: float) -> float:
    """Nearest bf16 value of x (ties to even), rounded once from fp64."""
    return float(_load().fo_round_bf16(float(x)))


def rope(x, pos, base: float, round_bf16: bool = False) -> np.ndarray:
    """Rotary position embedding (RoFormer, rotate-half pairing) of bf16 rows
    ``x`` [..., d] at positions ``pos`` (broadcast to x's leading shape; the
    layout's position ids). Returns fp64 [..., d]; with ``round_bf16`` each value
    is rounded once to bf16, the element type of rotated rows in a bf16 path."""
    lib = _load()
    xb = _bits(x)
    d = xb.shape[-1]
    lead = xb.shape[:-1]
    p = np.ascontiguousarray(np.broadcast_to(np.asarray(pos, dtype=np.int64), lead)).reshape(-1)
    n = p.size
    y = np.zeros((n, d), np.float64)
    lib.fo_rope(n, d, _ptr(p), float(base), int(round_bf16), _ptr(np.ascontiguousarray(xb.reshape(n, d))), _ptr(y))
    return y.reshape(xb.shape)


def attn_rows_f64(qf, kf, v, keep, win, scale: float, heads, rows):
    """``attn_rows`` with fp64 queries and keys (e.g. after ``rope``):
    qf/kf fp64 [n_heads, T, d], v bf16 [n_heads, T, d]."""
    lib = _load()
    qf = np.ascontiguousarray(qf, dtype=np.float64)
    kf = np.ascontiguousarray(kf, dtype=np.float64)
    vb = _bits(v)
    nh, T, d = qf.shape
    assert kf.shape == qf.shape and vb.shape == qf.shape
    keep = np.ascontiguousarray(keep, dtype=np.uint8)
    win = np.ascontiguousarray(win, dtype=np.int32)
    heads = np.ascontiguousarray(heads, dtype=np.int64)
    rows = np.ascontiguousarray(rows, dtype=np.int64)
    assert heads.shape == rows.shape
    n = rows.size
    o = np.zeros((n, d), np.float64)
    lse = np.zeros(n, np.float64)
    lib.fo_attn_rows_f64(T, d, _ptr(keep), _ptr(win), _ptr(qf), _ptr(kf), _ptr(vb), float(scale), n,
                         _ptr(heads), _ptr(rows), _ptr(o), _ptr(lse))
    return o, lse


def decode_f64(qf, knf, v_new, ring_kf, ring_v, R, win_kf, win_v, fill, scale: float):
    """``decode`` with fp64 queries and keys (rotated by the caller): qf/knf
    fp64 [n, d]; ring_kf fp64 [n, C_ring, d]; win_kf fp64 [n, C_win, d]; values
    bf16."""
    lib = _load()
    qf = np.ascontiguousarray(qf, dtype=np.float64)
    knf = np.ascontiguousarray(knf, dtype=np.float64)
    rkf = np.ascontiguousarray(ring_kf, dtype=np.float64)
    wkf = np.ascontiguousarray(win_kf, dtype=np.float64)
    vnb, rvb, wvb = _bits(v_new), _bits(ring_v), _bits(win_v)
    n, d = qf.shape
    R = np.ascontiguousarray(R, dtype=np.int64)
    fill = np.ascontiguousarray(fill, dtype=np.int64)
    assert (R <= rkf.shape[1]).all() and (fill < wkf.shape[1] + 1).all()
    o = np.zeros((n, d), np.float64)
    lse = np.zeros(n, np.float64)
    lib.fo_decode_f64(d, n, _ptr(rkf), _ptr(rvb), rkf.shape[1], _ptr(R), _ptr(wkf), _ptr(wvb), wkf.shape[1],
                      _ptr(fill), _ptr(qf), _ptr(knf), _ptr(vnb), float(scale), _ptr(o), _ptr(lse))
    return o, lse


def embed_tokens(tok, table_bits) -> np.ndarray:
    """Input rows of the augmented sequence (Sec. 3.2 "Setup and tokens": the
    FOCUS summary is a learned token inserted after each k-mer; App. A: each
    inserted token takes a position of its own): row i is the embedding-table row
    of token tok[i]. ``table_bits``: uint16 bf16 patterns [n_tokens, D]; returns
    the uint16 patterns [*tok.shape, D] (a lookup moves bits, nothing rounds).
    A token outside the table gives a zero row."""
    tok = np.asarray(tok)
    table = np.asarray(table_bits, dtype=np.uint16)
    out = np.zeros((*tok.shape, table.shape[1]), np.uint16)
    for idx in np.ndindex(*tok.shape):
        if int(tok[idx]) < table.shape[0]:
            out[idx] = table[int(tok[idx])]
    return out


def window_retained_rows(n: int, k: int, close_partial: bool = True, tail: int = 0) -> np.ndarray:
    """In-window augmented offsets of the rows KV retention keeps for a window
    of n bases with cadence k: its FOCUS rows and its last ``tail`` bases (App. A)."""
    lib = _load()
    cap = 2 * n + 2
    out = np.zeros(cap, np.int32)
    c = lib.fo_window_retained_rows(n, k, int(close_partial), int(tail), _ptr(out), cap)
    return out[:c]


def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to fp64 (used by tests to compare
    GPU bf16 outputs against fp64 oracle outputs)."""
    b = np.ascontiguousarray(bits, dtype=np.uint16).astype(np.uint32) << 16
    return b.view(np.float32).astype(np.float64)
