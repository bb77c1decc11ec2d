"""GPU parity of adaptive windowing (each window with its own length W_w and
cadence k_w; Sec. 5) against the fp64 oracle: the scheduled layout bit for bit,
masked-parallel and streaming prefill, the k-mer-local mask, and decode rolling
over windows of different lengths."""
import math

import numpy as np
import pytest
import torch

from oracle import focus_oracle as fo
from paper_2511_14694_gb300 import focus, inputs, pipeline
from test_gpu_parity import assert_attn_close, bits

pytestmark = pytest.mark.gpu

SCHEDULES = [
    # N, window lengths, cadences (both cycled to the window count), tail
    (2_500, [400, 1_000, 100, 1_000], [10, 25, 7, 200], 0),
    (1_037, [64, 1_000, 1_000], [8, 100, 3], 0),
    (3_000, [128, 64, 1_024, 16, 8, 52, 900, 700], [0, 5, 100, 1, 9, 13, 50, 1_000], 0),
    (3_000, [128, 64, 1_024, 16, 8, 52, 900, 700], [0, 5, 100, 1, 9, 13, 50, 1_000], 4),
    (20_000, [300, 1_700], [10, 100], 0),
]


@pytest.fixture(autouse=True)
def _clean_status():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    focus.device_status(clear=True)
    yield
    assert focus.device_status(clear=True) == 0, "a kernel reported an error"


def _sched(N, Ws, ks):
    Wfull = np.resize(np.asarray(Ws, np.int32), 4 * N // min(Ws) + 4)
    W = fo.window_schedule(N, Wfull)
    k = np.resize(np.asarray(ks, np.int32), W.size)
    return W, k


@pytest.mark.parametrize("N,Ws,ks,tail", SCHEDULES)
@pytest.mark.parametrize("close", [True, False])
def test_adaptive_layout_bit_exact(N, Ws, ks, tail, close):
    W, k = _sched(N, Ws, ks)
    nt = inputs.nucleotides(2, N, seed=5, device="cuda")
    L = focus.layout(N, W, k, nt=nt, close_tail=close, tail=tail)
    ref = fo.layout(N, W, k, nt=nt.cpu().numpy(), close_tail=close, tail=tail)
    assert (L["T"], L["R"], L["M"]) == (ref["T"], ref["R"], ref["M"])
    for name in ("kind", "src", "pos", "win", "keep", "win_off", "ring_off", "base_off", "tok"):
        assert np.array_equal(L[name].cpu().numpy(), ref[name]), name
    assert np.array_equal(L["sum_idx"].cpu().numpy(), ref["sum_idx"])


@pytest.mark.parametrize("N,Ws,ks,tail", SCHEDULES)
def test_adaptive_prefill_masked_parallel_matches_oracle(N, Ws, ks, tail):
    W, k = _sched(N, Ws, ks)
    B, H, d = 1, 2, 128
    L = focus.layout(N, W, k, tail=tail)
    q, kk, v = inputs.qkv((B, H, L["T"], d), seed=N + 1, device="cuda")
    cache = focus.Cache(B, H, d, C_ring=max(L["R"], 1))
    o, lse = pipeline.prefill_masked_parallel(cache, q, kk, v, L)
    torch.cuda.synchronize()
    ref = fo.layout(N, W, k, tail=tail)
    T = L["T"]
    o_ref, lse_ref = fo.attn_rows(q[0].cpu(), kk[0].cpu(), v[0].cpu(), ref["keep"], ref["win"], 1 / math.sqrt(d),
                                  np.repeat(np.arange(H), T), np.tile(np.arange(T), H))
    assert_attn_close(o, lse, o_ref.reshape(B, H, T, d), lse_ref.reshape(B, H, T), f"adaptive N={N}")
    assert np.array_equal(bits(cache.ring_k)[:, :, :L["R"]], bits(kk)[:, :, ref["sum_idx"]])


def test_adaptive_prefill_streaming_and_kmer_local():
    N, Ws, ks = 3_000, [128, 64, 1_024, 16, 8, 52, 900, 700], [0, 5, 100, 1, 9, 13, 50, 1_000]
    W, k = _sched(N, Ws, ks)
    B, H, d = 2, 1, 64
    L = focus.layout(N, W, k)
    q, kk, v = inputs.qkv((B, H, L["T"], d), seed=9, device="cuda")
    ref = fo.layout(N, W, k)
    T = L["T"]
    heads, rows = np.repeat(np.arange(B * H), T), np.tile(np.arange(T), B * H)
    flat = lambda t: t.reshape(B * H, T, d).cpu()  # noqa: E731
    for flags in (0, focus.PREFILL_KMER_LOCAL):
        cache = focus.Cache(B, H, d, C_ring=L["R"], k_sched=k)
        o = torch.empty_like(q)
        lse = torch.empty((B, H, T), dtype=torch.float32, device="cuda")
        off = L["win_off_host"]
        for w in range(L["M"]):
            a, e = int(off[w]), int(off[w + 1])
            sl = lambda t: t[:, :, a:e].contiguous()  # noqa: E731
            ow, lw = pipeline.prefill_window(cache, sl(q), sl(kk), sl(v), L, w, flags=flags)
            o[:, :, a:e] = ow
            lse[:, :, a:e] = lw
        torch.cuda.synchronize()
        if flags:
            km = fo.layout_kmer(N, W, k)
            o_ref, lse_ref = fo.attn_rows_kmer_local(flat(q), flat(kk), flat(v), ref["kind"], ref["win"], km,
                                                     1 / math.sqrt(d), heads, rows)
        else:
            o_ref, lse_ref = fo.attn_rows(flat(q), flat(kk), flat(v), ref["keep"], ref["win"], 1 / math.sqrt(d),
                                          heads, rows)
        assert_attn_close(o, lse, o_ref.reshape(B, H, T, d), lse_ref.reshape(B, H, T), f"adaptive flags={flags}")


def test_adaptive_kmer_tiled_prefill_matches_oracle():
    """Window lengths 700..1,200 and cadences 90..110 with the k-mer-local mask, at a
    size that selects the k-mer-tiled kernel (its tile count is the most any window
    needs, so the shorter windows carry empty tiles); ragged last window."""
    N, Ws, ks = 16_037, [700, 1_200, 900, 1_000], [90, 110, 100, 95, 105]
    W, k = _sched(N, Ws, ks)
    B, H, d = 1, 16, 64
    L = focus.layout(N, W, k)
    T = L["T"]
    q, kk, v = inputs.qkv((B, H, T, d), seed=17, device="cuda")
    cache = focus.Cache(B, H, d, C_ring=L["R"], k_sched=k)
    fl = focus.PREFILL_KMER_LOCAL
    assert focus.prefill_kernel(cache, q, kk, v, L, flags=fl) == "tcgen05 k-mer tiles"
    o, lse = pipeline.prefill_masked_parallel(cache, q, kk, v, L, flags=fl)
    torch.cuda.synchronize()
    ref = fo.layout(N, W, k)
    heads, rows = np.repeat(np.arange(H), T), np.tile(np.arange(T), H)
    o_ref, lse_ref = fo.attn_rows_kmer_local(q[0].cpu(), kk[0].cpu(), v[0].cpu(), ref["kind"], ref["win"],
                                             fo.layout_kmer(N, W, k), 1 / math.sqrt(d), heads, rows)
    assert_attn_close(o, lse, o_ref.reshape(B, H, T, d), lse_ref.reshape(B, H, T), "adaptive k-mer tiles")


def test_adaptive_decode_rolls_over_windows_of_different_lengths():
    """Decode with a per-window length schedule: each sequence fills its window
    to T_w = W_w + ceil(W_w / k_w) rows, then window-mode compaction keeps its
    FOCUS rows and moves on to the next window's length."""
    B, H, d = 3, 2, 64
    W_sched = np.array([20, 7, 33, 12, 5, 40, 9, 16], np.int32)
    k_sched = np.array([4, 3, 10, 12, 1, 7, 2, 5], np.int32)
    Tw = W_sched + -(-W_sched // k_sched)
    cache = focus.Cache(B, H, d, C_ring=256, C_win=int(Tw.max()) + 2, W=0, k_sched=k_sched, W_sched=W_sched)
    g = torch.Generator(device="cuda").manual_seed(8)
    for t in (cache.ring_k, cache.ring_v, cache.win_k, cache.win_v):
        t.copy_(torch.randn(t.shape, generator=g, device="cuda").bfloat16())
    R0, widx0, fill0 = np.array([0, 11, 40], np.int32), np.array([0, 1, 2], np.int32), np.array([0, 9, 30], np.int32)
    cache.ring_len.copy_(torch.from_numpy(R0))
    cache.win_idx.copy_(torch.from_numpy(widx0))
    cache.win_fill.copy_(torch.from_numpy(fill0))
    rk, rv = bits(cache.ring_k).copy(), bits(cache.ring_v).copy()
    wk, wv = bits(cache.win_k).copy(), bits(cache.win_v).copy()
    R, fill, widx = R0.copy(), fill0.copy(), widx0.copy()
    ws = cache.new_workspace()
    scale = 1 / math.sqrt(d)
    for step in range(90):
        q, kn, vn = inputs.qkv((B, H, d), seed=500 + step, device="cuda")
        o, lse = focus.attn_decode(cache, q, kn, vn, workspace=ws)
        focus.kv_compact_window(cache)
        qb, kb, vb = bits(q), bits(kn), bits(vn)
        o_ref, lse_ref = np.zeros((B, H, d)), np.zeros((B, H))
        for b in range(B):
            o_ref[b], lse_ref[b] = fo.decode(qb[b], kb[b], vb[b], rk[b], rv[b], [R[b]] * H, wk[b], wv[b],
                                             [fill[b]] * H, scale)
            wk[b, :, fill[b]], wv[b, :, fill[b]] = kb[b], vb[b]
            fill[b] += 1
            w = widx[b]
            if fill[b] == Tw[w]:
                keep_rows = fo.window_retained_rows(int(W_sched[w]), int(k_sched[w]), True, 0)
                rk[b, :, R[b]:R[b] + keep_rows.size] = wk[b][:, keep_rows]
                rv[b, :, R[b]:R[b] + keep_rows.size] = wv[b][:, keep_rows]
                R[b] += keep_rows.size
                fill[b] = 0
                widx[b] += 1
        assert_attn_close(o, lse, o_ref, lse_ref, f"adaptive decode step {step}")
    torch.cuda.synchronize()
    assert np.array_equal(cache.ring_len.cpu().numpy(), R)
    assert np.array_equal(cache.win_idx.cpu().numpy(), widx)
    assert np.array_equal(cache.win_fill.cpu().numpy(), fill)
    for b in range(B):
        assert np.array_equal(bits(cache.ring_k[b])[:, :R[b]], rk[b, :, :R[b]])
