"""GPU parity: the CUDA path (through the C ABI) against the fp64 oracle on the
same seeded inputs.

Bars: layout, position ids, gather indices and compaction are bit-exact.
Attention output O: max-abs <= 2e-2 and mean-abs <= 2e-3, and (because the
N(0,1)/sqrt(d) workloads give ~10x smaller outputs, where the absolute bars are
loose) relative RMS error <= 1e-2. LSE: |error| <= 1e-3 * max(1, |LSE|).
"""
import math

import numpy as np
import pytest
import torch

from oracle import focus_oracle as fo
from paper_2511_14694_gb300 import focus, inputs, pipeline

pytestmark = pytest.mark.gpu

O_MAX_ABS, O_MEAN_ABS, O_REL_RMS, LSE_REL = 2e-2, 2e-3, 1e-2, 1e-3


@pytest.fixture(autouse=True)
def _clean_status():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    focus.device_status(clear=True)
    yield
    assert focus.device_status(clear=True) == 0, "a kernel reported an error"


def assert_attn_close(o_gpu, lse_gpu, o_ref, lse_ref, what=""):
    og = o_gpu.detach().float().cpu().double().numpy().reshape(o_ref.shape)
    lg = lse_gpu.detach().cpu().double().numpy().reshape(lse_ref.shape)
    assert np.isfinite(og).all() and np.isfinite(lg).all(), what
    err = np.abs(og - o_ref)
    rel_rms = math.sqrt(float((err ** 2).mean())) / max(math.sqrt(float((o_ref ** 2).mean())), 1e-30)
    lerr = np.abs(lg - lse_ref) / np.maximum(1.0, np.abs(lse_ref))
    msg = f"{what}: max {err.max():.3e} mean {err.mean():.3e} relrms {rel_rms:.3e} lse {lerr.max():.3e}"
    assert err.max() <= O_MAX_ABS, msg
    assert err.mean() <= O_MEAN_ABS, msg
    assert rel_rms <= O_REL_RMS, msg
    assert lerr.max() <= LSE_REL, msg


def bits(t):
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


# ----------------------------------------------------------------------------- layout

LAYOUT_CASES = [
    (4_000, 1_000, [100], True), (128_000, 1_000, [100], True), (256_000, 1_000, [10, 25, 50, 100, 200], True),
    (1_000_000, 1_000, [100], True), (10, 4, [3], True), (1, 1, [1], True), (500, 1_000, [0], True),
    (77, 10, [20], True), (5_000, 1_024, [100], False), (5_000, 1_024, [100], True), (3_001, 3, [1, 2, 3, 4], False),
    (2_048, 2_048, [1], True),
]
TAIL_LAYOUT_CASES = [(4_000, 1_000, [100], True, 3), (3_001, 3, [1, 2, 3, 4], False, 1), (77, 10, [20], True, 10),
                     (5_000, 1_024, [100], False, 50), (500, 1_000, [0], True, 7), (10, 4, [3], True, 100)]


@pytest.mark.parametrize("N,W,ks,close,tail", [c + (0,) for c in LAYOUT_CASES] + TAIL_LAYOUT_CASES)
def test_layout_bit_exact(N, W, ks, close, tail):
    M = -(-N // W)
    k = inputs.k_schedule(M, ks, seed=N % 97)
    nt = inputs.nucleotides(2, N, seed=5, device="cuda")
    L = focus.layout(N, W, k, nt=nt, close_tail=close, tail=tail)
    ref = fo.layout(N, W, k, nt=nt.cpu().numpy(), close_tail=close, tail=tail)
    torch.cuda.synchronize()
    assert (L["T"], L["R"], L["M"]) == (ref["T"], ref["R"], ref["M"])
    for key in ("kind", "keep", "src", "pos", "win", "win_off", "ring_off", "sum_idx"):
        assert np.array_equal(L[key].cpu().numpy(), ref[key]), key
    assert np.array_equal(L["tok"].cpu().numpy(), ref["tok"])


# ----------------------------------------------------------------------------- prefill, masked-parallel

PREFILL_CASES = [
    # N, W, k schedule, B, H, d, std
    (4_000, 1_000, [100], 1, 4, 64, 1.0),            # 4 windows of 1 kb, k=100, the small parity workload
    (1_000, 300, [7], 2, 2, 128, 1.0),
    (777, 128, [1, 5, 50, 200], 1, 3, 64, 1.0),
    (500, 1_000, [0], 1, 2, 128, 1.0),                # compression disabled: plain causal
    (300, 64, [64], 1, 2, 64, 1.0),                   # T_w = 65: one row past a tile
    (20_000, 200, [10], 1, 2, 128, 1.0 / math.sqrt(128)),   # ring of up to 990 rows
    (3_333, 1_000, [3, 100, 1_000], 2, 1, 128, 1.0),  # ragged last window, k = W
]
TAIL_PREFILL_CASES = [
    # N, W, k schedule, B, H, d, std, tail
    (3_000, 500, [10, 50], 1, 2, 128, 1.0, 3),
    (1_000, 100, [7], 2, 1, 64, 1.0, 200),          # tail >= W: every row kept -> causal over all rows
    (4_100, 1_000, [100], 1, 2, 128, 1.0 / math.sqrt(128), 30),
]


# Ring capacity that sends the appendix-mask prefill to the one-CTA-per-item
# kernel: the persistent kernel serves only C_ring + max_rows <= 4,096 rows.
PER_ITEM_C_RING = 8_192


def _masked_parallel(N, W, ks, B, H, d, std, seed=0, flags=0, tail=0, c_ring=None):
    M = -(-N // W)
    k = inputs.k_schedule(M, ks, seed=seed + 1)
    L = focus.layout(N, W, k, tail=tail)
    q, kk, v = inputs.qkv((B, H, L["T"], d), std=std, seed=seed + 2, device="cuda")
    cache = focus.Cache(B, H, d, C_ring=c_ring or max(L["R"], 1))
    n = q.numel()
    canary = torch.full((n + 4096,), 7.0, dtype=torch.bfloat16, device="cuda")
    o = canary[:n].view(q.shape)
    o, lse = pipeline.prefill_masked_parallel(cache, q, kk, v, L, o=o, flags=flags)
    torch.cuda.synchronize()
    assert bool((canary[n:] == 7.0).all()), "prefill wrote past its output"
    return L, q, kk, v, cache, o, lse


@pytest.mark.parametrize("c_ring", [None, PER_ITEM_C_RING], ids=["persistent", "per_item"])
@pytest.mark.parametrize("N,W,ks,B,H,d,std,tail", [c + (0,) for c in PREFILL_CASES] + TAIL_PREFILL_CASES)
def test_prefill_masked_parallel_matches_oracle(N, W, ks, B, H, d, std, tail, c_ring):
    """Both tcgen05 kernels on the same inputs: a ring sized to the retained rows
    selects the persistent kernel for these short work items, a large ring the
    one-CTA-per-item kernel."""
    L, q, k, v, cache, o, lse = _masked_parallel(N, W, ks, B, H, d, std, seed=N, tail=tail, c_ring=c_ring)
    assert focus.prefill_kernel(cache, q, k, v, L) == ("tcgen05 persistent" if c_ring is None
                                                       else "tcgen05, one CTA per work item")
    ref_L = fo.layout(N, W, L["k_host"], tail=tail)
    T = L["T"]
    heads = np.repeat(np.arange(B * H), T)
    rows = np.tile(np.arange(T), B * H)
    o_ref, lse_ref = fo.attn_rows(q.reshape(B * H, T, d).cpu(), k.reshape(B * H, T, d).cpu(),
                                  v.reshape(B * H, T, d).cpu(), ref_L["keep"], ref_L["win"], 1.0 / math.sqrt(d),
                                  heads, rows)
    assert_attn_close(o, lse, o_ref.reshape(B, H, T, d), lse_ref.reshape(B, H, T), f"N={N} W={W} k={ks}")
    # compaction: ring == the FOCUS rows, bit for bit
    kb, vb = bits(k), bits(v)
    assert np.array_equal(bits(cache.ring_k)[:, :, :L["R"]], kb[:, :, ref_L["sum_idx"]])
    assert np.array_equal(bits(cache.ring_v)[:, :, :L["R"]], vb[:, :, ref_L["sum_idx"]])
    assert (cache.ring_len.cpu().numpy() == L["R"]).all()


def test_prefill_legacy_kernel_matches_oracle():
    N, W, ks, B, H, d = 2_000, 500, [50], 1, 2, 128
    L, q, k, v, cache, o, lse = _masked_parallel(N, W, ks, B, H, d, 1.0, seed=9, flags=focus.PREFILL_LEGACY_MMA)
    ref_L = fo.layout(N, W, L["k_host"])
    T = L["T"]
    o_ref, lse_ref = fo.attn_rows(q.reshape(H, T, d).cpu(), k.reshape(H, T, d).cpu(), v.reshape(H, T, d).cpu(),
                                  ref_L["keep"], ref_L["win"], 1.0 / math.sqrt(d), np.repeat(np.arange(H), T),
                                  np.tile(np.arange(T), H))
    assert_attn_close(o, lse, o_ref.reshape(B, H, T, d), lse_ref.reshape(B, H, T), "legacy")


# ----------------------------------------------------------------------------- prefill, k-mer-local mask (Sec. 3.2)

LOCAL_PREFILL_CASES = [
    # N, W, k schedule (cycled over the windows), B, H, d, std
    (4_000, 1_000, [100], 1, 2, 64, 1.0),
    (5_000, 1_024, [100], 1, 2, 128, 1.0),                   # partial k-mer closes every window
    (3_001, 300, [1, 7, 50, 0, 300, 1_000], 2, 1, 128, 1.0),  # k = 1 (300 FOCUS rows: 3 ring tiles), k = 0
                                                             # (no boundary for the next window), k >= W, ragged end
    (2_000, 2_000, [0], 1, 1, 64, 1.0),                      # one window, one k-mer: causal
    (20_000, 200, [10], 1, 2, 128, 1.0 / math.sqrt(128)),
    (300, 64, [64], 1, 2, 64, 1.0),                          # T_w = 65: one row past a tile
    (1_500, 700, [3, 128, 255], 1, 1, 64, 1.0),              # k-mers that straddle 128-row tiles
]


def _local_case(N, W, ks, B, H, d, std, seed):
    M = -(-N // W)
    k = np.resize(np.asarray(ks, np.int32), M)
    L = focus.layout(N, W, k)
    q, kk, v = inputs.qkv((B, H, L["T"], d), std=std, seed=seed, device="cuda")
    cache = focus.Cache(B, H, d, C_ring=max(L["R"], 1), k_sched=k)
    return L, k, q, kk, v, cache


def _local_ref(N, W, k, q, kk, v, heads, rows):
    B, H, T, d = q.shape
    ref_L = fo.layout(N, W, k)
    km = fo.layout_kmer(N, W, k)
    return fo.attn_rows_kmer_local(q.reshape(B * H, T, d).cpu(), kk.reshape(B * H, T, d).cpu(),
                                   v.reshape(B * H, T, d).cpu(), ref_L["kind"], ref_L["win"], km, 1.0 / math.sqrt(d),
                                   heads, rows)


# cases whose k-mers and visible ring rows fit one 128-row K/V tile, with at
# least 2,048 work items: the k-mer-tiled kernel runs when the host schedule is
# passed, the one-CTA-per-item kernel without it (and for the cases above)
LOCAL_TILED_CASES = [
    (16_000, 1_000, [100], 1, 32, 64, 1.0),                   # 10 one-k-mer tiles per window, RB = 16
    (5_000, 1_024, [100], 2, 32, 128, 1.0),                   # partial k-mer closes every window
    (20_000, 200, [10], 1, 16, 128, 1.0 / math.sqrt(128)),    # 9 k-mers per tile, RB = 24, ragged tiles
    (9_000, 1_000, [100, 50, 60], 1, 32, 128, 1.0),           # k per window: tiles of 1 or 2 k-mers, RB = 24;
                                                              # k = 60 gives the most tiles (17 of 61 rows)
]
LOCAL_TILED = {(N, W, B, H) for N, W, ks, B, H, *_ in LOCAL_TILED_CASES}


@pytest.mark.parametrize("host_schedule", [True, False])
@pytest.mark.parametrize("N,W,ks,B,H,d,std", LOCAL_PREFILL_CASES + LOCAL_TILED_CASES)
def test_prefill_kmer_local_matches_oracle(N, W, ks, B, H, d, std, host_schedule):
    L, k, q, kk, v, cache = _local_case(N, W, ks, B, H, d, std, seed=N + 7)
    fl = focus.PREFILL_KMER_LOCAL
    tiled = host_schedule and (N, W, B, H) in LOCAL_TILED
    want = "tcgen05 k-mer tiles" if tiled else "tcgen05, one CTA per work item"
    assert focus.prefill_kernel(cache, q, kk, v, L, flags=fl, host_schedule=host_schedule) == want
    n = q.numel()
    canary = torch.full((n + 4096,), 7.0, dtype=torch.bfloat16, device="cuda")
    o = canary[:n].view(q.shape)
    focus.kv_compact_bulk(cache, kk, v, L)
    o, lse = focus.attn_prefill(cache, q, kk, v, L, o=o, flags=fl, host_schedule=host_schedule)
    torch.cuda.synchronize()
    assert bool((canary[n:] == 7.0).all()), "prefill wrote past its output"
    T = L["T"]
    heads = np.repeat(np.arange(B * H), T)
    rows = np.tile(np.arange(T), B * H)
    o_ref, lse_ref = _local_ref(N, W, k, q, kk, v, heads, rows)
    assert_attn_close(o, lse, o_ref.reshape(B, H, T, d), lse_ref.reshape(B, H, T), f"local N={N} W={W} k={ks}")


@pytest.mark.parametrize("d", [64, 128])
def test_prefill_kmer_local_streaming_matches_oracle(d):
    """Window by window: compact window w into the ring, then prefill it."""
    N, W, ks, B, H = 3_000, 500, [10, 50, 0, 7, 100, 500], 2, 2
    L, k, q, kk, v, cache = _local_case(N, W, ks, B, H, d, 1.0, seed=31)
    o = torch.empty_like(q)
    lse = torch.empty((B, H, L["T"]), dtype=torch.float32, device="cuda")
    off = L["win_off_host"]
    for w in range(L["M"]):
        a, e = int(off[w]), int(off[w + 1])
        sl = lambda t: t[:, :, a:e].contiguous()  # noqa: E731
        ow, lw = pipeline.prefill_window(cache, sl(q), sl(kk), sl(v), L, w, flags=focus.PREFILL_KMER_LOCAL)
        o[:, :, a:e] = ow
        lse[:, :, a:e] = lw
    torch.cuda.synchronize()
    T = L["T"]
    heads = np.repeat(np.arange(B * H), T)
    rows = np.tile(np.arange(T), B * H)
    o_ref, lse_ref = _local_ref(N, W, k, q, kk, v, heads, rows)
    assert_attn_close(o, lse, o_ref.reshape(B, H, T, d), lse_ref.reshape(B, H, T), "local streaming")


def test_prefill_kmer_local_argument_checks():
    N, W = 1_000, 500
    L, k, q, kk, v, cache = _local_case(N, W, [10], 1, 1, 64, 1.0, seed=1)
    bad_tail = focus.Cache(1, 1, 64, C_ring=L["R"], k_sched=k, tail=2)
    with pytest.raises(RuntimeError, match="unsupported"):
        focus.attn_prefill(bad_tail, q, kk, v, L, flags=focus.PREFILL_KMER_LOCAL)
    no_k = focus.Cache(1, 1, 64, C_ring=L["R"])          # k schedule of one window, two needed
    with pytest.raises(RuntimeError, match="invalid"):
        focus.attn_prefill(no_k, q, kk, v, L, flags=focus.PREFILL_KMER_LOCAL)
    with pytest.raises(RuntimeError, match="unsupported"):
        focus.attn_prefill(cache, q, kk, v, L, flags=focus.PREFILL_KMER_LOCAL | focus.PREFILL_LEGACY_MMA)
    with pytest.raises(RuntimeError, match="invalid"):
        focus.attn_prefill(cache, q, kk, v, L, flags=8)


# ----------------------------------------------------------------------------- prefill, sequential / streaming

@pytest.mark.parametrize("d,tail", [(64, 0), (128, 0), (128, 5)])
def test_prefill_streaming_matches_sequential_oracle(d, tail):
    N, W, ks, B, H = 3_000, 500, [10, 50, 100, 7], 2, 2
    M = -(-N // W)
    k_s = inputs.k_schedule(M, ks, seed=4)
    L = focus.layout(N, W, k_s, tail=tail)
    q, k, v = inputs.qkv((B, H, L["T"], d), seed=21, device="cuda")
    cache = focus.Cache(B, H, d, C_ring=L["R"])
    o = torch.empty_like(q)
    lse = torch.empty((B, H, L["T"]), dtype=torch.float32, device="cuda")
    off = L["win_off_host"]
    for w in range(M):
        a, e = int(off[w]), int(off[w + 1])
        sl = lambda t: t[:, :, a:e].contiguous()  # noqa: E731
        ow, lw = pipeline.prefill_window(cache, sl(q), sl(k), sl(v), L, w)
        o[:, :, a:e] = ow
        lse[:, :, a:e] = lw
    torch.cuda.synchronize()
    ref_L = fo.layout(N, W, k_s, tail=tail)
    for b in range(B):
        for h in range(H):
            o_ref, lse_ref, rk, rv = fo.prefill_sequential(q[b, h].cpu(), k[b, h].cpu(), v[b, h].cpu(),
                                                           ref_L["win_off"], ref_L["keep"], 1.0 / math.sqrt(d))
            assert_attn_close(o[b, h], lse[b, h], o_ref, lse_ref, f"stream b={b} h={h}")
            assert np.array_equal(bits(cache.ring_k[b, h, :L["R"]]), rk)
            assert np.array_equal(bits(cache.ring_v[b, h, :L["R"]]), rv)


@pytest.mark.parametrize("d,tail,flags", [(128, 0, 0), (64, 3, 0), (128, 0, focus.PREFILL_KMER_LOCAL)])
def test_prefill_streaming_overlapped_equals_sequential(d, tail, flags):
    """pipeline.prefill_streaming (compaction first, consecutive windows' attention
    overlapping on two streams; one window or a chunk of windows per attention
    call) gives, bit for bit, the outputs and ring of the one-window-at-a-time loop
    (which the test above pins to the oracle)."""
    N, W, ks, B, H = 3_000, 500, [10, 50, 100, 7], 2, 2
    M = -(-N // W)
    k_s = inputs.k_schedule(M, ks, seed=4)
    L = focus.layout(N, W, k_s, tail=tail)
    q, k, v = inputs.qkv((B, H, L["T"], d), seed=23, device="cuda")
    off = L["win_off_host"]
    win = lambda t, w: t[:, :, int(off[w]):int(off[w + 1])].contiguous()  # noqa: E731
    c_seq = focus.Cache(B, H, d, C_ring=L["R"], k_sched=k_s, tail=tail)
    seq = [pipeline.prefill_window(c_seq, win(q, w), win(k, w), win(v, w), L, w, flags=flags) for w in range(M)]
    c_ovl = focus.Cache(B, H, d, C_ring=L["R"], k_sched=k_s, tail=tail)
    qkv_w = [(win(q, w), win(k, w), win(v, w)) for w in range(M)]
    outs = [torch.empty_like(x[0]) for x in qkv_w]
    lses = [torch.empty(x[0].shape[:3], dtype=torch.float32, device="cuda") for x in qkv_w]
    pipeline.prefill_streaming(c_ovl, L, lambda w: qkv_w[w], outs, lses, flags=flags)
    torch.cuda.synchronize()
    for w in range(M):
        assert np.array_equal(bits(outs[w]), bits(seq[w][0])), f"window {w}"
        assert torch.equal(lses[w], seq[w][1]), f"window {w}"
    assert np.array_equal(bits(c_ovl.ring_k), bits(c_seq.ring_k))
    assert np.array_equal(bits(c_ovl.ring_v), bits(c_seq.ring_v))
    # chunks of windows per attention call (each window still compacted on its own):
    # the same items on the same kernel, so the same bits
    for chunk in (2, 4):
        c_chk = focus.Cache(B, H, d, C_ring=L["R"], k_sched=k_s, tail=tail)
        spn = lambda t, w0, w1: t[:, :, int(off[w0]):int(off[w1])].contiguous()  # noqa: E731
        spans = {w0: (spn(q, w0, min(w0 + chunk, M)), spn(k, w0, min(w0 + chunk, M)), spn(v, w0, min(w0 + chunk, M)))
                 for w0 in range(0, M, chunk)}
        outs = [torch.empty_like(spans[w0][0]) for w0 in range(0, M, chunk)]
        lses = [torch.empty(x.shape[:3], dtype=torch.float32, device="cuda") for x in outs]
        pipeline.prefill_streaming(c_chk, L, lambda w0, w1: spans[w0], outs, lses, flags=flags, chunk=chunk)
        torch.cuda.synchronize()
        for n, w0 in enumerate(range(0, M, chunk)):
            for w in range(w0, min(w0 + chunk, M)):
                a, e = int(off[w] - off[w0]), int(off[w + 1] - off[w0])
                assert np.array_equal(bits(outs[n][:, :, a:e]), bits(seq[w][0])), f"chunk {chunk} window {w}"
                assert torch.equal(lses[n][:, :, a:e], seq[w][1]), f"chunk {chunk} window {w}"
        assert np.array_equal(bits(c_chk.ring_k), bits(c_seq.ring_k))
        assert np.array_equal(bits(c_chk.ring_v), bits(c_seq.ring_v))


@pytest.mark.parametrize("d,flags,rope,chunk,g", [(128, 0, 0.0, 3, 1), (64, 0, 0.0, 1, 1),
                                                  (128, focus.PREFILL_KMER_LOCAL, 0.0, 4, 1),
                                                  (128, 0, 10_000.0, 2, 1), (64, 0, 0.0, 2, 4)])
def test_prefill_streaming_graph_equals_eager(d, flags, rope, chunk, g):
    """pipeline.StreamingGraph (the streaming step captured once as a CUDA graph)
    replays to the eager pipeline.prefill_streaming's outputs and ring, bit for
    bit, and rewrites them on every replay (outputs and ring are cleared between
    replays); chunk 3 leaves a partial last chunk, the rotary case allocates its
    workspaces before the capture, g = 4 groups the query heads."""
    N, W, ks, B, H = 6_000, 500, [10, 50, 100, 7], 2, 2
    M = -(-N // W)
    k_s = inputs.k_schedule(M, ks, seed=5)
    L = focus.layout(N, W, k_s)
    q = inputs.normal_bf16((B, H * g, L["T"], d), 1.0, seed=29, device="cuda")
    k, v = (inputs.normal_bf16((B, H, L["T"], d), 1.0, seed=s, device="cuda") for s in (30, 31))
    off = L["win_off_host"]
    spn = lambda t, w0, w1: t[:, :, int(off[w0]):int(off[w1])].contiguous()  # noqa: E731
    spans = {w0: tuple(spn(t, w0, min(w0 + chunk, M)) for t in (q, k, v)) for w0 in range(0, M, chunk)}
    qkv = (lambda w0: spans[w0]) if chunk == 1 else (lambda w0, w1: spans[w0])
    runs = {}
    for mode in ("eager", "graph"):
        cache = focus.Cache(B, H, d, C_ring=L["R"], k_sched=k_s, rope_theta=rope, q_per_kv=g)
        outs = [torch.empty_like(spans[w0][0]) for w0 in range(0, M, chunk)]
        lses = [torch.empty(x.shape[:3], dtype=torch.float32, device="cuda") for x in outs]
        if mode == "eager":
            pipeline.prefill_streaming(cache, L, qkv, outs, lses, flags=flags, chunk=chunk)
        else:
            g = pipeline.StreamingGraph(cache, L, qkv, outs, lses, flags=flags, chunk=chunk)
            for _ in range(2):
                for t in outs + lses + [cache.ring_k, cache.ring_v]:
                    t.zero_()
                g.replay()
        torch.cuda.synchronize()
        runs[mode] = (outs, lses, cache)
    (o_e, l_e, c_e), (o_g, l_g, c_g) = runs["eager"], runs["graph"]
    for n in range(len(o_e)):
        assert np.array_equal(bits(o_g[n]), bits(o_e[n])), f"call {n}"
        assert torch.equal(l_g[n], l_e[n]), f"call {n}"
    assert np.array_equal(bits(c_g.ring_k), bits(c_e.ring_k))
    assert np.array_equal(bits(c_g.ring_v), bits(c_e.ring_v))


# ----------------------------------------------------------------------------- decode

class DecodeModel:
    """Host mirror of the decode cache evolved with the oracle's rules (App. A.2)."""

    def __init__(self, ring_k, ring_v, R, win_k, win_v, fill, widx, W, k_sched, tail=0):
        self.rk, self.rv = bits(ring_k).copy(), bits(ring_v).copy()
        self.wk, self.wv = bits(win_k).copy(), bits(win_v).copy()
        self.R, self.fill, self.widx = R.copy(), fill.copy(), widx.copy()
        self.W, self.k, self.tail = W, np.asarray(k_sched), tail

    def step(self, q, kn, vn, scale):
        B, H, d = q.shape
        qb, kb, vb = bits(q), bits(kn), bits(vn)
        o = np.zeros((B, H, d))
        lse = np.zeros((B, H))
        for b in range(B):
            oo, ll = fo.decode(qb[b], kb[b], vb[b], self.rk[b], self.rv[b], [self.R[b]] * H, self.wk[b], self.wv[b],
                               [self.fill[b]] * H, scale)
            o[b], lse[b] = oo, ll
            f = self.fill[b]
            self.wk[b, :, f], self.wv[b, :, f] = kb[b], vb[b]
            self.fill[b] += 1
            kw = int(self.k[self.widx[b]])
            Tw = self.W + (-(-self.W // kw) if kw > 0 else 0)
            if self.fill[b] == Tw:                       # window complete: retain its FOCUS rows
                rows = fo.window_retained_rows(self.W, kw, True, self.tail)
                r = self.R[b]
                self.rk[b, :, r:r + rows.size] = self.wk[b][:, rows]
                self.rv[b, :, r:r + rows.size] = self.wv[b][:, rows]
                self.R[b] += rows.size
                self.fill[b] = 0
                self.widx[b] += 1
        return o, lse


@pytest.mark.parametrize("d,tail", [(64, 0), (128, 0), (128, 4)])
def test_decode_steps_match_oracle(d, tail):
    B, H, W = 3, 2, 50
    k_sched = np.array([10, 7, 25, 50, 3, 10, 10, 10], np.int32)
    C_ring, C_win = 512, 72
    cache = focus.Cache(B, H, d, C_ring=C_ring, C_win=C_win, W=W, k_sched=k_sched, tail=tail)
    g = torch.Generator(device="cuda").manual_seed(3)
    for t in (cache.ring_k, cache.ring_v, cache.win_k, cache.win_v):
        t.copy_(torch.randn(t.shape, generator=g, device="cuda").bfloat16())
    R0 = np.array([0, 37, 300], np.int32)
    widx0 = np.array([0, 1, 2], np.int32)
    fill0 = np.array([0, 50, 20], np.int32)   # window 1 has T_w = 58
    cache.ring_len.copy_(torch.from_numpy(R0))
    cache.win_idx.copy_(torch.from_numpy(widx0))
    cache.win_fill.copy_(torch.from_numpy(fill0))
    model = DecodeModel(cache.ring_k, cache.ring_v, R0, cache.win_k, cache.win_v, fill0, widx0, W, k_sched, tail)
    ws = cache.new_workspace()
    scale = 1.0 / math.sqrt(d)
    for step in range(70):
        q, kn, vn = inputs.qkv((B, H, d), seed=100 + step, device="cuda")
        o, lse = focus.attn_decode(cache, q, kn, vn, workspace=ws)
        focus.kv_compact_window(cache)
        o_ref, lse_ref = model.step(q, kn, vn, scale)
        assert_attn_close(o, lse, o_ref, lse_ref, f"decode step {step}")
    torch.cuda.synchronize()
    assert np.array_equal(cache.ring_len.cpu().numpy(), model.R)
    assert np.array_equal(cache.win_fill.cpu().numpy(), model.fill)
    assert np.array_equal(cache.win_idx.cpu().numpy(), model.widx)
    for b in range(B):
        assert np.array_equal(bits(cache.ring_k[b])[:, :model.R[b]], model.rk[b, :, :model.R[b]])
        assert np.array_equal(bits(cache.ring_v[b])[:, :model.R[b]], model.rv[b, :, :model.R[b]])


def test_decode_full_window_is_reported_not_trapped():
    B, H, d, W = 1, 1, 64, 10
    cache = focus.Cache(B, H, d, C_ring=16, C_win=11, W=W, k_sched=[10])
    cache.win_fill.fill_(11)                      # T_w = 11: already full
    q, kn, vn = inputs.qkv((B, H, d), seed=1, device="cuda")
    focus.attn_decode(cache, q, kn, vn)
    assert focus.device_status(clear=True) == 3   # FOCUS_ERR_CAPACITY
    assert int(cache.win_fill[0]) == 11


def test_layout_empty_sequence():
    L = focus.layout(0, 1_000, [100])
    assert (L["T"], L["R"], L["M"]) == (0, 0, 0)
    assert L["win_off_host"].tolist() == [0] and L["ring_off_host"].tolist() == [0]


def test_bulk_compaction_overflow_is_reported_not_trapped():
    N, W, H, d = 4_000, 1_000, 2, 64
    L = focus.layout(N, W, [100])
    cache = focus.Cache(1, H, d, C_ring=L["R"] - 1)
    k = inputs.normal_bf16((1, H, L["T"], d), 1.0, seed=3, device="cuda")
    v = inputs.normal_bf16((1, H, L["T"], d), 1.0, seed=4, device="cuda")
    focus.kv_compact_bulk(cache, k, v, L)
    assert focus.device_status(clear=True) == 3   # FOCUS_ERR_CAPACITY
    assert int(cache.ring_len[0]) == 0
    assert not cache.ring_k.any()


# ----------------------------------------------------------------------------- full-size workloads, sampled rows

def _sample_rows(L, n_windows, rows_per_window, seed):
    rng = np.random.default_rng(seed)
    M = L["M"]
    ws = sorted(set([0, M - 1] + list(rng.integers(0, M, size=n_windows - 2))))
    off = L["win_off_host"]
    rows = []
    for w in ws:
        a, e = int(off[w]), int(off[w + 1])
        rows += [a, e - 1] + list(rng.integers(a, e, size=rows_per_window - 2))
    return np.array(sorted(set(rows)), np.int64)


@pytest.mark.parametrize("name", ["prefill_128kb_h32_d128", "prefill_256kb_ksweep_h32_d128", "causal_128kb_h32_d128"])
def test_full_size_prefill_sampled(name):
    """Full-size launches (the persistent kernel at 128 kb, the one-CTA-per-item
    kernel on the 256 kb k sweep and on plain causal attention over 128 kb, whose
    longest work item runs 1,000 K/V tiles) on sampled rows against the oracle."""
    from paper_2511_14694_gb300.workloads import WORKLOADS
    cfg = WORKLOADS[name]
    N, W, B, H, d = cfg["N"], cfg["W"], cfg["B"], cfg["H"], cfg["d"]
    M = -(-N // W)
    k_s = inputs.k_schedule(M, cfg["k"], seed=inputs.DEFAULT_SEED)
    L = focus.layout(N, W, k_s)
    q, k, v = inputs.qkv((B, H, L["T"], d), std=cfg["std"], seed=inputs.DEFAULT_SEED, device="cuda")
    cache = focus.Cache(B, H, d, C_ring=L["R"])
    o, lse = pipeline.prefill_masked_parallel(cache, q, k, v, L)
    torch.cuda.synchronize()
    rows = _sample_rows(L, 6, 4 if L["M"] > 1 else 24, seed=1)
    heads = [0, 7, 31]
    ref_L = fo.layout(N, W, k_s)
    o_ref, lse_ref = fo.attn_rows(q[0, heads].cpu(), k[0, heads].cpu(), v[0, heads].cpu(), ref_L["keep"],
                                  ref_L["win"], 1.0 / math.sqrt(d), np.repeat(np.arange(len(heads)), rows.size),
                                  np.tile(rows, len(heads)))
    og = o[0, heads][:, rows]
    lg = lse[0, heads][:, rows]
    assert_attn_close(og, lg, o_ref.reshape(len(heads), rows.size, d), lse_ref.reshape(len(heads), rows.size), name)
    assert (cache.ring_len.cpu().numpy() == L["R"]).all()


def test_full_size_decode_sampled():
    """Batch 64, 32 heads, d=128, 10,000 retained summaries + partly filled windows
    (fill ~ U{0..1009}); three steps, sequences at fill 1009 roll their window."""
    from paper_2511_14694_gb300.workloads import WORKLOADS
    cfg = WORKLOADS["decode_1mb_b64_h32_d128"]
    B, H, d, W, R = cfg["B"], cfg["H"], cfg["d"], cfg["W"], cfg["R"]
    k_sched = np.full(2_000, cfg["k"][0], np.int32)
    T_w = W + W // cfg["k"][0]
    cache = focus.Cache(B, H, d, C_ring=R + 256, C_win=1_024, W=W, k_sched=k_sched)
    for i, t in enumerate((cache.ring_k, cache.ring_v, cache.win_k, cache.win_v)):
        t.copy_(inputs.normal_bf16(t.shape, cfg["std"], seed=50 + i, device="cuda"))
    fill0 = inputs.start_fill(B, T_w - 1, seed=inputs.DEFAULT_SEED)
    fill0[:4] = T_w - 1
    cache.ring_len.fill_(R)
    cache.win_idx.fill_(R // (W // cfg["k"][0]))
    cache.win_fill.copy_(torch.from_numpy(fill0))
    rng = np.random.default_rng(0)
    pairs = [(0, 0), (1, 5), (3, 31)] + [(int(b), int(h)) for b, h in zip(rng.integers(0, B, 9), rng.integers(0, H, 9))]
    ws = cache.new_workspace()
    for step in range(3):
        R_now = cache.ring_len.cpu().numpy().copy()
        fill_now = cache.win_fill.cpu().numpy().copy()
        snap = {(b, h): (cache.ring_k[b, h].cpu(), cache.ring_v[b, h].cpu(), cache.win_k[b, h].cpu(),
                         cache.win_v[b, h].cpu()) for b, h in pairs}
        q, kn, vn = inputs.qkv((B, H, d), std=cfg["std"], seed=200 + step, device="cuda")
        o, lse = focus.attn_decode(cache, q, kn, vn, workspace=ws)
        focus.kv_compact_window(cache)
        torch.cuda.synchronize()
        for b, h in pairs:
            rk, rv, wk, wv = snap[(b, h)]
            o_ref, lse_ref = fo.decode(q[b, h][None].cpu(), kn[b, h][None].cpu(), vn[b, h][None].cpu(), rk[None],
                                       rv[None], [R_now[b]], wk[None], wv[None], [fill_now[b]], 1.0 / math.sqrt(d))
            assert_attn_close(o[b, h][None], lse[b, h][None], o_ref, lse_ref, f"decode b={b} h={h} step={step}")
    assert (cache.ring_len.cpu().numpy()[:4] == R + W // cfg["k"][0]).all()
    assert (cache.win_fill.cpu().numpy()[:4] == 2).all()


def test_full_size_streaming_sampled():
    """Batch 4, N = 1 Mb, W = 1,000, k = 100, 32 heads, d = 128: one prefill call and
    one compaction per window (App. A.2). Sampled windows of two heads are checked
    against the oracle's sequential form; the final ring (10,000 rows) bit-exactly."""
    from paper_2511_14694_gb300.workloads import WORKLOADS
    cfg = WORKLOADS["stream_1mb_b4_h32_d128"]
    B, N, W, H, d, P = cfg["B"], cfg["N"], cfg["W"], cfg["H"], cfg["d"], cfg["pool"]
    M = -(-N // W)
    L = focus.layout(N, W, [cfg["k"][0]])
    off = L["win_off_host"]
    Tw = int(off[1] - off[0])
    pq, pk, pv = inputs.qkv((P, B, H, Tw, d), std=cfg["std"], seed=inputs.DEFAULT_SEED, device="cuda")
    cache = focus.Cache(B, H, d, C_ring=L["R"])
    want = [0, 1, 437, 998, 999]
    b, heads = 1, [0, 17]
    got = {}
    for w in range(M):
        o, lse = pipeline.prefill_window(cache, pq[w % P], pk[w % P], pv[w % P], L, w)
        if w in want:
            got[w] = (o[b, heads].cpu(), lse[b, heads].cpu())
    torch.cuda.synchronize()
    assert (cache.ring_len.cpu().numpy() == L["R"]).all()
    ref_L = fo.layout(N, W, [cfg["k"][0]])
    want_mask = np.zeros(M, np.uint8)
    want_mask[want] = 1
    for i, h in enumerate(heads):
        full = [torch.cat([t[w % P, b, h] for w in range(M)]).cpu() for t in (pq, pk, pv)]
        o_ref, lse_ref, rk, rv = fo.prefill_sequential(*full, ref_L["win_off"], ref_L["keep"], 1.0 / math.sqrt(d),
                                                       want=want_mask)
        for w in want:
            a, e = int(off[w]), int(off[w + 1])
            assert_attn_close(got[w][0][i], got[w][1][i], o_ref[a:e], lse_ref[a:e], f"stream w={w} h={h}")
        assert np.array_equal(bits(cache.ring_k[b, h]), rk)
        assert np.array_equal(bits(cache.ring_v[b, h]), rv)


# ----------------------------------------------------------------------------- full-size: the extra modes, sampled rows

def test_full_size_kmer_local_prefill_sampled():
    """128 kb, 32 heads, d = 128, k-mer-local mask (Sec. 3.2), in the launch
    configuration the bench times; sampled rows of three heads."""
    from paper_2511_14694_gb300.workloads import WORKLOADS
    cfg = WORKLOADS["prefill_128kb_h32_d128"]
    N, W, B, H, d = cfg["N"], cfg["W"], cfg["B"], cfg["H"], cfg["d"]
    M = -(-N // W)
    k_s = inputs.k_schedule(M, cfg["k"], seed=inputs.DEFAULT_SEED)
    L = focus.layout(N, W, k_s)
    q, k, v = inputs.qkv((B, H, L["T"], d), std=cfg["std"], seed=inputs.DEFAULT_SEED, device="cuda")
    cache = focus.Cache(B, H, d, C_ring=L["R"], k_sched=k_s)
    o, lse = pipeline.prefill_masked_parallel(cache, q, k, v, L, flags=focus.PREFILL_KMER_LOCAL)
    torch.cuda.synchronize()
    rows = _sample_rows(L, 6, 4, seed=2)
    heads = [0, 13, 31]
    ref_L = fo.layout(N, W, k_s)
    km = fo.layout_kmer(N, W, k_s)
    o_ref, lse_ref = fo.attn_rows_kmer_local(q[0, heads].cpu(), k[0, heads].cpu(), v[0, heads].cpu(), ref_L["kind"],
                                             ref_L["win"], km, 1.0 / math.sqrt(d),
                                             np.repeat(np.arange(len(heads)), rows.size), np.tile(rows, len(heads)))
    assert_attn_close(o[0, heads][:, rows], lse[0, heads][:, rows], o_ref.reshape(len(heads), rows.size, d),
                      lse_ref.reshape(len(heads), rows.size), "full-size k-mer-local")


def test_full_size_rope_prefill_sampled():
    """128 kb, 32 heads, d = 128, rotary base 500,000 (positions up to 129,279):
    sampled rows of two heads against the oracle's fp64 rotation rounded to bf16."""
    from paper_2511_14694_gb300.workloads import WORKLOADS
    cfg = WORKLOADS["prefill_128kb_h32_d128"]
    N, W, B, H, d, theta = cfg["N"], cfg["W"], cfg["B"], cfg["H"], cfg["d"], 500_000.0
    L = focus.layout(N, W, cfg["k"])
    q, k, v = inputs.qkv((B, H, L["T"], d), std=cfg["std"], seed=inputs.DEFAULT_SEED, device="cuda")
    cache = focus.Cache(B, H, d, C_ring=L["R"], rope_theta=theta)
    o, lse = pipeline.prefill_masked_parallel(cache, q, k, v, L)
    torch.cuda.synchronize()
    rows = _sample_rows(L, 5, 4, seed=3)
    heads = [0, 21]
    ref_L = fo.layout(N, W, cfg["k"])
    pos = np.arange(L["T"])
    qf = fo.rope(q[0, heads].cpu(), pos, theta, round_bf16=True)
    kf = fo.rope(k[0, heads].cpu(), pos, theta, round_bf16=True)
    o_ref, lse_ref = fo.attn_rows_f64(qf, kf, v[0, heads].cpu(), ref_L["keep"], ref_L["win"], 1.0 / math.sqrt(d),
                                      np.repeat(np.arange(len(heads)), rows.size), np.tile(rows, len(heads)))
    assert_attn_close(o[0, heads][:, rows], lse[0, heads][:, rows], o_ref.reshape(len(heads), rows.size, d),
                      lse_ref.reshape(len(heads), rows.size), "full-size rope")


def test_full_size_gqa_decode_sampled():
    """Batch 64, 32 query heads over 8 K/V heads (q_per_kv = 4), d = 128, 10,000
    retained rows + partly filled windows: two steps, sampled query heads."""
    from paper_2511_14694_gb300.workloads import WORKLOADS
    cfg = WORKLOADS["decode_1mb_b64_h32_d128"]
    B, Hq, d, W, R, g = cfg["B"], cfg["H"], cfg["d"], cfg["W"], cfg["R"], 4
    H = Hq // g
    kk = cfg["k"][0]
    Tw = W + W // kk
    cache = focus.Cache(B, H, d, C_ring=R + 256, C_win=1_024, W=W, k_sched=np.full(2_000, kk, np.int32), q_per_kv=g)
    for i, t in enumerate((cache.ring_k, cache.ring_v, cache.win_k, cache.win_v)):
        t.copy_(inputs.normal_bf16(t.shape, cfg["std"], seed=60 + i, device="cuda"))
    fill0 = inputs.start_fill(B, Tw - 1, seed=inputs.DEFAULT_SEED)
    cache.ring_len.fill_(R)
    cache.win_idx.fill_(R // (W // kk))
    cache.win_fill.copy_(torch.from_numpy(fill0))
    ws = cache.new_workspace()
    pairs = [(0, 0), (5, 3), (17, 31), (63, 12)]
    for step in range(2):
        R_now, fill_now = cache.ring_len.cpu().numpy().copy(), cache.win_fill.cpu().numpy().copy()
        snap = {(b, hq): tuple(x[b, hq // g].cpu() for x in (cache.ring_k, cache.ring_v, cache.win_k, cache.win_v))
                for b, hq in pairs}
        q = inputs.normal_bf16((B, Hq, d), cfg["std"], seed=210 + step, device="cuda")
        kn, vn = (inputs.normal_bf16((B, H, d), cfg["std"], seed=220 + 2 * step + i, device="cuda") for i in (0, 1))
        o, lse = focus.attn_decode(cache, q, kn, vn, workspace=ws)
        focus.kv_compact_window(cache)
        torch.cuda.synchronize()
        for b, hq in pairs:
            rk, rv, wk, wv = snap[(b, hq)]
            o_ref, lse_ref = fo.decode(q[b, hq][None].cpu(), kn[b, hq // g][None].cpu(), vn[b, hq // g][None].cpu(),
                                       rk[None], rv[None], [R_now[b]], wk[None], wv[None], [fill_now[b]],
                                       1.0 / math.sqrt(d))
            assert_attn_close(o[b, hq][None], lse[b, hq][None], o_ref, lse_ref, f"gqa decode b={b} hq={hq}")
