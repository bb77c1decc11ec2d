"""CPU checks of the C-ABI library: it builds, loads, exports every function
include/focus.h declares, its struct layouts match the binding's, and its
host-only logic (layout sizes, argument validation) is right. No kernel is
launched here."""
import ctypes
import os
import re

import numpy as np
import pytest

from oracle import focus_oracle as fo
from paper_2511_14694_gb300 import focus, inputs

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "focus.h")


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:const\s+)?[A-Za-z_][A-Za-z0-9_]*\s*\*?\s*(focus_[a-z_0-9]+)\s*\(", src,
                                 flags=re.M)))


def test_library_exports_every_declared_function():
    lib = focus.load()
    names = declared_functions()
    assert {"focus_layout", "focus_attn_prefill", "focus_attn_decode", "focus_kv_compact"} <= set(names)
    for n in names:
        assert hasattr(lib, n), f"{n} declared in focus.h but not exported"


def test_struct_sizes_match_c_layout():
    # 2 x int64 + 8 pointers; 8 pointers + 7 int32 (+pad); see focus.h
    assert ctypes.sizeof(focus.LayoutOut) == 16 + 10 * 8
    assert ctypes.sizeof(focus.CacheDesc) == 8 * 8 + 8 * 4 + 8 + 8 + 8 + 8
    assert ctypes.sizeof(focus.PrefillArgs) == 5 * 8 + 8 + 2 * 8 + 6 * 4 + 2 * 8 + 8
    assert ctypes.sizeof(focus.CompactArgs) == 2 * 8 + 2 * 8 + 2 * 8 + 3 * 4 + 4
    # 12 buffer pointers, n_nt, W (+pad), d_W_sched, n_windows (+pad), d_k_sched, flags, tail, layout,
    # max_rows, scale, prefill_flags (+pad), workspace, its size, groups (+pad), two streams
    assert ctypes.sizeof(focus.PrefillHostArgs) == 12 * 8 + 8 + 8 + 8 + 8 + 8 + 8 + 8 + 16 + 8 + 8 + 8 + 16


def test_version_and_status_strings():
    lib = focus.load()
    assert lib.focus_version() >= 100
    for code in range(7):
        assert lib.focus_status_string(code)


@pytest.mark.parametrize("N,W,ks,close,tail", [(4_000, 1_000, [100], True, 0), (128_000, 1_000, [100], True, 0),
                                               (5_000, 1_024, [100], False, 0), (10, 4, [3], True, 0),
                                               (256_000, 1_000, [10, 25, 50, 100, 200], True, 0),
                                               (77, 100, [0], True, 0), (4_000, 1_000, [100], True, 4),
                                               (77, 10, [3], False, 20)])
def test_layout_size_matches_oracle(N, W, ks, close, tail):
    M = -(-N // W)
    k = inputs.k_schedule(M, ks, seed=1)
    T, R, M2, mx = focus.layout_size(N, W, k, close_tail=close, tail=tail)
    To, Ro, Mo = fo.layout_size(N, W, k, close_tail=close, tail=tail)
    assert (T, R, M2) == (To, Ro, Mo)
    L = fo.layout(N, W, k, close_tail=close, tail=tail)
    assert mx == int(np.diff(L["win_off"]).max())


def test_host_validation_rejects_bad_arguments():
    lib = focus.load()
    T = ctypes.c_int64()
    k = np.array([100], np.int32)
    # wrong window count, negative N, missing schedule
    assert lib.focus_layout_size(1000, 1000, 2, k.ctypes.data, 1, 0, ctypes.byref(T), None, None) == 1
    assert lib.focus_layout_size(-1, 1000, 0, k.ctypes.data, 1, 0, ctypes.byref(T), None, None) == 1
    assert lib.focus_layout_size(1000, 1000, 1, None, 1, 0, ctypes.byref(T), None, None) == 1
    assert lib.focus_layout_size(1000, 0, 1, k.ctypes.data, 1, 0, ctypes.byref(T), None, None) == 1
    assert lib.focus_layout_size(1000, 1000, 1, k.ctypes.data, 1, -1, ctypes.byref(T), None, None) == 1
    neg = np.array([-3], np.int32)
    assert lib.focus_layout_size(1000, 1000, 1, neg.ctypes.data, 1, 0, ctypes.byref(T), None, None) == 1
    # null descriptors
    assert lib.focus_attn_prefill(None, None, None) == 1
    assert lib.focus_kv_compact(None, None, None) == 1
    assert lib.focus_attn_decode(None, None, None, None, 1.0, None, None, None, 0, None) == 1
    # unsupported head dim is rejected before any CUDA call
    c = focus.CacheDesc()
    c.B, c.H, c.d, c.C_ring = 1, 1, 96, 0
    a = focus.PrefillArgs()
    assert lib.focus_attn_prefill(ctypes.byref(c), ctypes.byref(a), None) == 2
    c.d = 128
    # null q/k/v
    assert lib.focus_attn_prefill(ctypes.byref(c), ctypes.byref(a), None) == 1
    assert lib.focus_decode_workspace_size(None) == 0


def test_layout_size_edge_cases():
    lib = focus.load()
    T, R, mx = ctypes.c_int64(-1), ctypes.c_int64(-1), ctypes.c_int32(-1)
    # empty sequence: M = 0, nothing to lay out
    assert lib.focus_layout_size(0, 1000, 0, None, 1, 0, ctypes.byref(T), ctypes.byref(R), ctypes.byref(mx)) == 0
    assert (T.value, R.value, mx.value) == (0, 0, 0)
    # single base, single window
    k = np.array([1], np.int32)
    assert lib.focus_layout_size(1, 1, 1, k.ctypes.data, 1, 0, ctypes.byref(T), ctypes.byref(R), None) == 0
    assert (T.value, R.value) == (2, 1)
    # an augmented length beyond int32 offsets is refused, not truncated
    M = 2_000
    kk = np.ones(M, np.int32)
    assert lib.focus_layout_size(2_000_000_000, 1_000_000, M, kk.ctypes.data, 1, 0, ctypes.byref(T), None,
                                 None) == 2


def test_prefill_flag_checks_need_no_gpu():
    """Flag validation happens on the host before any CUDA call (T_span = 0 makes
    a valid call a no-op)."""
    lib = focus.load()
    c = focus.CacheDesc()
    c.B, c.H, c.d, c.C_ring = 1, 1, 64, 0
    a = focus.PrefillArgs()
    a.q = a.k = a.v = a.o = 4096
    a.d_win_off = a.d_ring_off = 4096
    a.n_windows, a.w_begin, a.w_end, a.max_rows, a.scale, a.T_span = 2, 0, 2, 10, 0.125, 0
    call = lambda flags: (setattr(a, "flags", flags), lib.focus_attn_prefill(ctypes.byref(c), ctypes.byref(a), None))[1]  # noqa: E731
    assert call(0) == 0
    assert call(focus.PREFILL_LEGACY_MMA) == 0
    assert call(8) == 1                                                   # unknown flag bit
    assert call(focus.PREFILL_KMER_LOCAL) == 1                            # no k schedule
    c.k_per_window, c.n_windows = 4096, 1
    assert call(focus.PREFILL_KMER_LOCAL) == 1                            # schedule shorter than w_end
    c.n_windows = 2
    assert call(focus.PREFILL_KMER_LOCAL) == 0
    assert call(focus.PREFILL_KMER_LOCAL | focus.PREFILL_LEGACY_MMA) == 2
    c.tail = 1
    assert call(focus.PREFILL_KMER_LOCAL) == 2                            # boundary tails not supported


def test_prefill_kernel_choice_needs_no_gpu():
    """focus_prefill_kernel names the kernel focus_attn_prefill would launch: the
    persistent tcgen05 kernel for the appendix mask without the rotary embedding
    while C_ring + max_rows <= 4,096, the one-CTA-per-item kernel otherwise, the
    legacy kernel on request; arguments are checked as for the launch."""
    lib = focus.load()
    c = focus.CacheDesc()
    c.B, c.H, c.d = 1, 2, 128
    c.ring_k = c.ring_v = 4096                        # never dereferenced: the query touches no memory
    a = focus.PrefillArgs()
    a.q = a.k = a.v = a.o = 4096
    a.d_win_off = a.d_ring_off = 4096
    a.n_windows, a.w_begin, a.w_end, a.scale, a.T_span = 128, 0, 128, 0.125, 129_280

    def choice(C_ring, max_rows, flags=0):
        c.C_ring, a.max_rows, a.flags = C_ring, max_rows, flags
        out = ctypes.c_int32(-1)
        rc = lib.focus_prefill_kernel(ctypes.byref(c), ctypes.byref(a), ctypes.byref(out))
        return rc, out.value

    assert choice(1_280, 1_010) == (0, 2)            # 128 windows of 1 kb, k = 100: short items
    assert choice(3_086, 1_010) == (0, 2)            # exactly 4,096 rows
    assert choice(3_087, 1_010) == (0, 1)
    assert choice(10_000, 1_010) == (0, 1)           # a long ring
    assert choice(1, 128_000) == (0, 1)              # one long window
    assert choice(1_280, 1_010, focus.PREFILL_LEGACY_MMA) == (0, 0)
    c.k_per_window, c.n_windows = 4096, 128
    assert choice(1_280, 1_010, focus.PREFILL_KMER_LOCAL) == (0, 1)       # no host schedule
    ks = np.full(128, 100, np.int32)
    a.h_k_per_window = ks.ctypes.data
    assert choice(1_280, 1_010, focus.PREFILL_KMER_LOCAL) == (0, 3)       # k-mers of 101 rows, <= 12 ring rows
    ks[5] = 10                                                            # ~100 ring rows in a tile: too many
    assert choice(1_280, 1_010, focus.PREFILL_KMER_LOCAL) == (0, 1)
    ks[5] = 150                                                           # a k-mer of 151 rows: too long
    assert choice(1_280, 1_010, focus.PREFILL_KMER_LOCAL) == (0, 1)
    ks[5] = 50                                                            # 21 ring rows: RB = 24, 104-row k-mer room
    assert choice(1_280, 1_010, focus.PREFILL_KMER_LOCAL) == (0, 3)
    a.h_k_per_window = None
    c.rope_theta = 10_000.0
    assert choice(1_280, 1_010) == (0, 1)            # rotary embedding without a workspace
    # with the workspace focus_prefill_workspace_size asks for (per-head counters,
    # then the span's q and k, rotated there by a pass): the kernel the arguments
    # take without the embedding
    c.C_ring, a.max_rows, a.flags = 1_280, 1_010, 0
    need = lib.focus_prefill_workspace_size(ctypes.byref(c), ctypes.byref(a))
    assert need == 256 + c.B * c.H * 2 * a.T_span * c.d * 2
    a.workspace, a.workspace_bytes = 4096, need
    rp = focus.PREFILL_KERNEL_ROTATION_PASS
    assert choice(1_280, 1_010) == (0, rp | 2)
    a.workspace_bytes = need - 1
    assert choice(1_280, 1_010) == (0, 1)            # too small: the per-item kernel rotating its tiles
    a.workspace, a.workspace_bytes = 4100, need
    assert choice(1_280, 1_010)[0] == 2              # misaligned workspace
    a.workspace, a.workspace_bytes = 4096, need
    assert choice(10_000, 1_010) == (0, rp | 1)      # long items: the per-item kernel, on the rotated rows
    assert lib.focus_prefill_workspace_size(ctypes.byref(c), ctypes.byref(a)) == need
    a.h_k_per_window = ks.ctypes.data
    # the k-mer-tiled kernel rotates its tiles in place: no pass, no workspace
    assert choice(1_280, 1_010, focus.PREFILL_KMER_LOCAL) == (0, 3)
    assert lib.focus_prefill_workspace_size(ctypes.byref(c), ctypes.byref(a)) == 0
    a.workspace, a.workspace_bytes = None, 0
    assert choice(1_280, 1_010, focus.PREFILL_KMER_LOCAL) == (0, 3)
    a.flags = 0
    a.workspace, a.workspace_bytes = 4096, need
    a.h_k_per_window = None
    # grouped-query heads on short items: the persistent kernel rotates into the
    # workspace itself (counters + q of the 4 query heads and k of each K/V head)
    c.q_per_kv = 4
    need4 = lib.focus_prefill_workspace_size(ctypes.byref(c), ctypes.byref(a))
    assert need4 == 256 + c.B * c.H * 5 * a.T_span * c.d * 2
    a.workspace_bytes = need4
    assert choice(1_280, 1_010) == (0, 2)            # no pass: the persistent kernel rotates
    assert choice(10_000, 1_010) == (0, rp | 1)
    c.q_per_kv = 1
    a.workspace, a.workspace_bytes = None, 0
    assert choice(1_280, 1_010, focus.PREFILL_LEGACY_MMA)[0] == 2      # legacy has no rotary embedding
    c.rope_theta = 0.0
    assert lib.focus_prefill_workspace_size(ctypes.byref(c), ctypes.byref(a)) == 0
    assert choice(1_280, 1_010, 8)[0] == 1                              # unknown flag bit
    assert lib.focus_prefill_kernel(ctypes.byref(c), ctypes.byref(a), None) == 1


def test_rope_argument_checks_need_no_gpu():
    """A negative or non-finite rotary base is refused on the host; decode with
    the rotary embedding needs pos_base."""
    lib = focus.load()
    c = focus.CacheDesc()
    c.B, c.H, c.d, c.C_ring = 1, 1, 64, 0
    a = focus.PrefillArgs()
    a.q = a.k = a.v = a.o = 4096
    a.d_win_off = a.d_ring_off = 4096
    a.n_windows, a.w_begin, a.w_end, a.max_rows, a.scale, a.T_span = 1, 0, 1, 10, 0.125, 0
    for bad in (-1.0, float("nan"), float("inf")):
        c.rope_theta = bad
        assert lib.focus_attn_prefill(ctypes.byref(c), ctypes.byref(a), None) == 1
    c.rope_theta = 10_000.0
    assert lib.focus_attn_prefill(ctypes.byref(c), ctypes.byref(a), None) == 0
    a.flags = focus.PREFILL_LEGACY_MMA                        # the legacy kernel has no rotation
    assert lib.focus_attn_prefill(ctypes.byref(c), ctypes.byref(a), None) == 2
    a.flags = 0
    c.win_k = c.win_v = c.ring_len = c.win_fill = c.win_idx = c.k_per_window = 4096
    c.W, c.n_windows, c.C_win = 10, 1, 16
    assert lib.focus_attn_decode(ctypes.byref(c), 4096, 4096, 4096, ctypes.c_float(0.125), 4096, None, 4096,
                                 1 << 20, None) == 1
    assert lib.focus_attn_decode_noalloc(ctypes.byref(c), 4096, 4096, 4096, ctypes.c_float(0.125), 4096, None,
                                         None) == 1


@pytest.mark.parametrize("N,Ws,ks,tail", [(2_500, [400, 1_000, 100, 1_000], [10, 25, 7, 200], 0),
                                          (1_037, [64, 1_000, 1_000], [8, 100, 3], 5),
                                          (300, [128, 64, 32, 16, 8, 52], [0, 5, 32, 1, 9, 13], 2)])
def test_layout_size_sched_matches_oracle(N, Ws, ks, tail):
    T, R, M, mx = focus.layout_size(N, Ws, ks[:len(fo.window_schedule(N, Ws))], tail=tail)
    L = fo.layout(N, Ws, ks[:M], tail=tail)
    assert (T, R, M) == (L["T"], L["R"], L["M"])
    assert mx == int(np.diff(L["win_off"]).max())


def test_layout_size_sched_rejects_bad_schedules():
    lib = focus.load()
    T = ctypes.c_int64()
    k = np.array([5, 5, 5], np.int32)
    for Ws, M in (([30, 30], 2), ([30, 0, 80], 3), ([60, 50, 10], 3), ([40, 50], 2)):
        w = np.array(Ws, np.int32)
        assert lib.focus_layout_size_sched(100, M, w.ctypes.data, k.ctypes.data, 1, 0, ctypes.byref(T), None,
                                           None) == 1, Ws
    w = np.array([30, 30, 40], np.int32)
    assert lib.focus_layout_size_sched(100, 3, w.ctypes.data, k.ctypes.data, 1, 0, ctypes.byref(T), None, None) == 0
    assert lib.focus_layout_size_sched(100, 3, None, k.ctypes.data, 1, 0, ctypes.byref(T), None, None) == 1


def test_cache_part_checks_contiguity():
    """Cache.part views a contiguous part of the cache: all heads of a range of
    sequences, or a head range of one sequence (no device needed)."""
    c = focus.Cache(2, 4, 64, C_ring=16, device="cpu")
    p = c.part(h0=1, h1=3, b0=1, b1=2)
    assert (p.desc.B, p.desc.H) == (1, 2)
    assert p.desc.ring_k == c.ring_k.data_ptr() + (1 * 4 + 1) * 16 * 64 * 2
    assert p.desc.ring_len == c.ring_len.data_ptr() + 4
    assert c.part(b0=1).desc.B == 1
    with pytest.raises(ValueError):
        c.part(h0=1, h1=3)                        # two sequences x a head range: not contiguous
    with pytest.raises(ValueError):
        c.part(b0=2)


def test_embed_tokens_argument_checks_need_no_gpu():
    """focus_embed_tokens refuses bad widths and tables on the host; no rows is a
    no-op that touches no pointer."""
    lib = focus.load()
    call = lambda n_rows, tab, n_tok, D, out: lib.focus_embed_tokens(4096, n_rows, tab, n_tok, D, out, None)  # noqa: E731
    assert call(0, None, 5, 64, None) == 0                   # nothing to do
    assert call(10, 4096, 0, 64, 4096) == 1                  # empty table
    assert call(10, 4096, 257, 64, 4096) == 1                # token ids are bytes
    assert call(10, 4096, 5, 0, 4096) == 1
    assert call(10, 4096, 5, 12, 4096) == 2                  # D not a multiple of 8
    assert call(10, 4104, 5, 64, 4096) == 2                  # table not 16-byte aligned
    assert call(10, 4096, 5, 64, 4100) == 2                  # out not 16-byte aligned
    assert call(-1, 4096, 5, 64, 4096) == 1
    assert lib.focus_embed_tokens(None, 10, 4096, 5, 64, 4096, None) == 1


def test_selftest_timeout_argument_checks_need_no_gpu():
    """The failure-path self-test refuses a zero or over-long wait on the host."""
    lib = focus.load()
    assert lib.focus_selftest_timeout(0, None) == 1
    assert lib.focus_selftest_timeout(10_000_000_001, None) == 1


def test_cache_snapshot_restore_round_trip():
    """A snapshot holds copies of the whole cache state and restores it in place."""
    c = focus.Cache(2, 1, 64, C_ring=8, C_win=4, W=3, k_sched=[2], device="cpu")
    c.ring_k.fill_(1.0)
    c.win_fill.fill_(2)
    snap = c.snapshot()
    assert set(snap) == {"ring_k", "ring_v", "win_k", "win_v", "ring_len", "win_fill", "win_idx", "pos_base"}
    c.ring_k.fill_(3.0)
    c.win_fill.fill_(0)
    c.restore(snap)
    assert bool((c.ring_k == 1.0).all()) and bool((c.win_fill == 2).all())


def test_decode_bindings_check_head_counts_before_any_call(monkeypatch):
    # q must have H * q_per_kv heads and k_new/v_new H: a mismatch is a ValueError
    # raised on the host, before the library is called (a short q or o would be
    # read or written past its end by the kernels)
    import torch

    class NoLib:
        def __getattr__(self, name):
            raise AssertionError(f"{name} called despite mismatched heads")

    monkeypatch.setattr(focus, "load", lambda: NoLib())
    monkeypatch.setattr(focus, "_cuda", lambda t, name, dtype=None: t)
    cache = type("C", (), {"H": 4, "q_per_kv": 4})()
    q = torch.zeros((2, 4, 128), dtype=torch.bfloat16)         # should be 16 query heads
    kv = torch.zeros((2, 4, 128), dtype=torch.bfloat16)
    for fn in (focus.attn_decode_noalloc, focus.attn_decode):
        with pytest.raises(ValueError, match="heads"):
            fn(cache, q, kv, kv)
    with pytest.raises(ValueError, match="heads"):
        focus.attn_decode_noalloc(cache, torch.zeros((2, 16, 128)), kv[:, :2], kv)


@pytest.mark.parametrize("N,W", [(0, 1_000), (1, 1), (4_000, 1_000), (4_001, 1_000), (128_000, 1_000), (77, 100),
                                 (1_000_000, 1_000), (10, 4)])
def test_layout_windows_matches_oracle(N, W):
    lib = focus.load()
    M = ctypes.c_int32(-1)
    assert lib.focus_layout_windows(N, W, ctypes.byref(M)) == 0
    assert M.value == fo.n_windows(N, W) == len(fo.window_schedule(N, W))


@pytest.mark.parametrize("N,Ws", [(0, [5]), (10, [10]), (10, [3, 3, 3, 3, 3]), (9, [3, 3, 3, 3]),
                                  (1_000, [400, 100, 700, 1]), (5, [1, 1, 1, 1, 1, 9, 9])])
def test_layout_windows_sched_matches_oracle(N, Ws):
    lib = focus.load()
    W = np.asarray(Ws, np.int32)
    M = ctypes.c_int32(-1)
    assert lib.focus_layout_windows_sched(N, W.size, W.ctypes.data, ctypes.byref(M)) == 0
    assert M.value == len(fo.window_schedule(N, W))
    assert np.array_equal(focus.window_lengths(N, W), fo.window_schedule(N, W))


def test_layout_windows_rejects_bad_arguments():
    lib = focus.load()
    M = ctypes.c_int32()
    assert lib.focus_layout_windows(-1, 10, ctypes.byref(M)) == 1
    assert lib.focus_layout_windows(10, 0, ctypes.byref(M)) == 1
    assert lib.focus_layout_windows(10, 10, None) == 1
    short = np.array([3, 3], np.int32)
    assert lib.focus_layout_windows_sched(7, 2, short.ctypes.data, ctypes.byref(M)) == 1     # does not cover
    bad = np.array([3, 0, 9], np.int32)
    assert lib.focus_layout_windows_sched(7, 3, bad.ctypes.data, ctypes.byref(M)) == 1       # empty window
    assert lib.focus_layout_windows_sched(7, 3, None, ctypes.byref(M)) == 1
    with pytest.raises(focus.FocusError):
        focus.window_lengths(7, short)


def test_prefill_host_rejects_bad_arguments_before_any_cuda_call():
    lib = focus.load()
    c = focus.CacheDesc()
    c.B, c.H, c.d = 1, 2, 128
    L = focus.LayoutOut()
    a = focus.PrefillHostArgs()
    for f in ("h_nt", "h_q", "h_k", "h_v", "h_o", "d_nt", "d_q", "d_k", "d_v", "d_o"):
        setattr(a, f, 4096)
    a.layout = ctypes.pointer(L)
    a.n_nt, a.W, a.n_windows, a.groups = 1_000, 1_000, 1, 2
    a.copy_in, a.copy_out = 8, 16
    assert lib.focus_prefill_host(None, ctypes.byref(a), 24) == 1
    a.groups = 0
    assert lib.focus_prefill_host(ctypes.byref(c), ctypes.byref(a), 24) == 1       # groups < 1
    a.groups = 2
    assert lib.focus_prefill_host(ctypes.byref(c), ctypes.byref(a), 8) == 1        # copy_in is the stream
    a.copy_out = 8
    assert lib.focus_prefill_host(ctypes.byref(c), ctypes.byref(a), 24) == 1       # one copy stream for both
    a.copy_out, a.h_lse = 16, 4096
    assert lib.focus_prefill_host(ctypes.byref(c), ctypes.byref(a), 24) == 1       # lse out without a device lse
    a.h_lse, a.d_q = None, None
    assert lib.focus_prefill_host(ctypes.byref(c), ctypes.byref(a), 24) == 1       # missing device buffer


def test_binding_constants_match_the_header():
    """The binding's flag, token and kernel constants are the header's #defines."""
    src = open(HEADER).read()
    defs = {m[0]: int(m[1]) for m in re.findall(r"^#define (FOCUS_[A-Z_]+) (\d+)u?\s*$", src, re.M)}
    assert defs["FOCUS_SUMMARY_TOKEN"] == focus.SUMMARY_TOKEN
    assert defs["FOCUS_LAYOUT_CLOSE_TAIL"] == focus.LAYOUT_CLOSE_TAIL
    assert defs["FOCUS_PREFILL_LEGACY_MMA"] == focus.PREFILL_LEGACY_MMA
    assert defs["FOCUS_PREFILL_KMER_LOCAL"] == focus.PREFILL_KMER_LOCAL
    assert defs["FOCUS_PREFILL_KERNEL_ROTATION_PASS"] == focus.PREFILL_KERNEL_ROTATION_PASS
    names = {"FOCUS_PREFILL_KERNEL_LEGACY": "legacy mma.sync", "FOCUS_PREFILL_KERNEL_PER_ITEM":
             "tcgen05, one CTA per work item", "FOCUS_PREFILL_KERNEL_PERSISTENT": "tcgen05 persistent",
             "FOCUS_PREFILL_KERNEL_KMER": "tcgen05 k-mer tiles"}
    for define, name in names.items():
        assert focus.PREFILL_KERNELS[defs[define]] == name
    assert all(not defs["FOCUS_PREFILL_KERNEL_ROTATION_PASS"] & k for k in focus.PREFILL_KERNELS)  # a bit of its own
