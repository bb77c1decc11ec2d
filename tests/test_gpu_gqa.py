"""GPU parity of grouped-query heads (q_per_kv = g query heads share each K/V
head; query head hq reads K/V head hq // g) against the fp64 oracle, which sees
each query head with its K/V head's rows: masked-parallel, streaming and
k-mer-local prefill, the rotary embedding, and decode for every grouping the
decode kernel specialises (one, two or four query heads per K/V pass)."""
import math

import numpy as np
import pytest
import torch

from oracle import focus_oracle as fo
from paper_2511_14694_gb300 import focus, inputs, pipeline
from test_gpu_parity import PER_ITEM_C_RING, assert_attn_close, bits

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _clean_status():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    focus.device_status(clear=True)
    yield
    assert focus.device_status(clear=True) == 0, "a kernel reported an error"


def _expand(x, g):
    """[B, H, ...] -> [B, H * g, ...]: each K/V head repeated for its query heads."""
    return x.repeat_interleave(g, dim=1)


@pytest.mark.parametrize("g,d,flags,rope,c_ring", [(2, 128, 0, 0.0, None), (4, 64, 0, 0.0, None),
                                                   (8, 128, 0, 0.0, None), (3, 64, 0, 0.0, None),
                                                   (4, 128, 0, 0.0, PER_ITEM_C_RING), (3, 64, 0, 0.0, PER_ITEM_C_RING),
                                                   (4, 128, "local", 0.0, None), (2, 128, 0, 10_000.0, None)])
def test_gqa_prefill_masked_parallel_matches_oracle(g, d, flags, rope, c_ring):
    """A ring sized to the retained rows selects the persistent kernel for the
    appendix mask; PER_ITEM_C_RING the one-CTA-per-item kernel (which also serves
    the k-mer-local mask and the rotary embedding)."""
    N, W, ks, B, H = 5_000, 1_000, [100, 10, 50, 100, 7], 1, 2
    k = np.resize(np.asarray(ks, np.int32), 5)
    L = focus.layout(N, W, k)
    T = L["T"]
    q = inputs.normal_bf16((B, H * g, T, d), 1.0, seed=1, device="cuda")
    kk, v = (inputs.normal_bf16((B, H, T, d), 1.0, seed=s, device="cuda") for s in (2, 3))
    cache = focus.Cache(B, H, d, C_ring=c_ring or L["R"], k_sched=k, q_per_kv=g, rope_theta=rope)
    fl = focus.PREFILL_KMER_LOCAL if flags == "local" else 0
    # the rotary embedding takes the persistent kernel too, with the workspace the binding allocates
    persistent = c_ring is None and not fl
    assert focus.prefill_kernel(cache, q, kk, v, L, flags=fl) == ("tcgen05 persistent" if persistent
                                                                  else "tcgen05, one CTA per work item")
    o, lse = pipeline.prefill_masked_parallel(cache, q, kk, v, L, flags=fl)
    torch.cuda.synchronize()
    assert o.shape == q.shape and lse.shape == (B, H * g, T)
    ref = fo.layout(N, W, k)
    Hq = H * g
    heads, rows = np.repeat(np.arange(Hq), T), np.tile(np.arange(T), Hq)
    qh, kh, vh = q[0].cpu(), _expand(kk, g)[0].cpu(), _expand(v, g)[0].cpu()
    if rope:
        pos = np.arange(T)
        o_ref, lse_ref = fo.attn_rows_f64(fo.rope(qh, pos, rope, round_bf16=True),
                                          fo.rope(kh, pos, rope, round_bf16=True), vh, ref["keep"], ref["win"],
                                          1 / math.sqrt(d), heads, rows)
    elif fl:
        o_ref, lse_ref = fo.attn_rows_kmer_local(qh, kh, vh, ref["kind"], ref["win"], fo.layout_kmer(N, W, k),
                                                 1 / math.sqrt(d), heads, rows)
    else:
        o_ref, lse_ref = fo.attn_rows(qh, kh, vh, ref["keep"], ref["win"], 1 / math.sqrt(d), heads, rows)
    assert_attn_close(o, lse, o_ref.reshape(B, Hq, T, d), lse_ref.reshape(B, Hq, T), f"gqa g={g} d={d} {flags}")
    if not rope:     # the ring holds the K/V heads' FOCUS rows, once per K/V head
        assert np.array_equal(bits(cache.ring_k)[:, :, :L["R"]], bits(kk)[:, :, ref["sum_idx"]])


def test_gqa_kmer_tiled_prefill_matches_oracle():
    """The k-mer-local mask at a size that selects the k-mer-tiled kernel (16 windows
    x 10 tiles x 16 query heads = 2,560 items, above its 2,048-item threshold), with
    four query heads per K/V head and a ragged last window; every row is checked."""
    N, W, k_, B, H, g, d = 16_037, 1_000, 100, 1, 4, 4, 64
    k = np.full(-(-N // W), k_, np.int32)
    L = focus.layout(N, W, k)
    T = L["T"]
    q = inputs.normal_bf16((B, H * g, T, d), 1.0, seed=31, device="cuda")
    kk, v = (inputs.normal_bf16((B, H, T, d), 1.0, seed=s, device="cuda") for s in (32, 33))
    cache = focus.Cache(B, H, d, C_ring=L["R"], k_sched=k, q_per_kv=g)
    fl = focus.PREFILL_KMER_LOCAL
    assert focus.prefill_kernel(cache, q, kk, v, L, flags=fl) == "tcgen05 k-mer tiles"
    o, lse = pipeline.prefill_masked_parallel(cache, q, kk, v, L, flags=fl)
    torch.cuda.synchronize()
    ref = fo.layout(N, W, k)
    Hq = H * g
    heads, rows = np.repeat(np.arange(Hq), T), np.tile(np.arange(T), Hq)
    o_ref, lse_ref = fo.attn_rows_kmer_local(q[0].cpu(), _expand(kk, g)[0].cpu(), _expand(v, g)[0].cpu(),
                                             ref["kind"], ref["win"], fo.layout_kmer(N, W, k), 1 / math.sqrt(d),
                                             heads, rows)
    assert_attn_close(o, lse, o_ref.reshape(B, Hq, T, d), lse_ref.reshape(B, Hq, T), "gqa k-mer tiles")


def test_gqa_prefill_streaming_matches_oracle():
    N, W, ks, B, H, g, d = 3_000, 500, [10, 50, 0, 7, 100, 500], 2, 2, 4, 64
    k = np.resize(np.asarray(ks, np.int32), 6)
    L = focus.layout(N, W, k)
    T = L["T"]
    q = inputs.normal_bf16((B, H * g, T, d), 1.0, seed=4, device="cuda")
    kk, v = (inputs.normal_bf16((B, H, T, d), 1.0, seed=s, device="cuda") for s in (5, 6))
    cache = focus.Cache(B, H, d, C_ring=L["R"], q_per_kv=g)
    o = torch.empty_like(q)
    lse = torch.empty((B, H * g, T), dtype=torch.float32, device="cuda")
    off = L["win_off_host"]
    for w in range(L["M"]):
        a, e = int(off[w]), int(off[w + 1])
        sl = lambda t: t[:, :, a:e].contiguous()  # noqa: E731
        ow, lw = pipeline.prefill_window(cache, sl(q), sl(kk), sl(v), L, w)
        o[:, :, a:e] = ow
        lse[:, :, a:e] = lw
    torch.cuda.synchronize()
    ref = fo.layout(N, W, k)
    Hq = H * g
    flat = lambda t: t.reshape(B * Hq, T, d).cpu()  # noqa: E731
    heads, rows = np.repeat(np.arange(B * Hq), T), np.tile(np.arange(T), B * Hq)
    o_ref, lse_ref = fo.attn_rows(flat(q), flat(_expand(kk, g)), flat(_expand(v, g)), ref["keep"], ref["win"],
                                  1 / math.sqrt(d), heads, rows)
    assert_attn_close(o, lse, o_ref.reshape(B, Hq, T, d), lse_ref.reshape(B, Hq, T), "gqa streaming")


@pytest.mark.parametrize("g,d", [(1, 64), (2, 128), (3, 64), (4, 128), (8, 64), (8, 128)])
def test_gqa_decode_steps_match_oracle(g, d):
    B, H, W = 3, 2, 50
    k_sched = np.array([10, 7, 25, 50, 3, 10, 10, 10], np.int32)
    cache = focus.Cache(B, H, d, C_ring=512, C_win=72, W=W, k_sched=k_sched, q_per_kv=g)
    gen = torch.Generator(device="cuda").manual_seed(11)
    for t in (cache.ring_k, cache.ring_v, cache.win_k, cache.win_v):
        t.copy_(torch.randn(t.shape, generator=gen, device="cuda").bfloat16())
    R0, widx0, fill0 = np.array([0, 37, 300], np.int32), np.array([0, 1, 2], np.int32), np.array([0, 50, 20], np.int32)
    cache.ring_len.copy_(torch.from_numpy(R0))
    cache.win_idx.copy_(torch.from_numpy(widx0))
    cache.win_fill.copy_(torch.from_numpy(fill0))
    rk, rv = bits(cache.ring_k).copy(), bits(cache.ring_v).copy()
    wk, wv = bits(cache.win_k).copy(), bits(cache.win_v).copy()
    R, fill, widx = R0.copy(), fill0.copy(), widx0.copy()
    ws = cache.new_workspace()
    scale = 1 / math.sqrt(d)
    Hq = H * g
    for step in range(40):
        q = inputs.normal_bf16((B, Hq, d), 1.0, seed=700 + step, device="cuda")
        kn, vn = (inputs.normal_bf16((B, H, d), 1.0, seed=900 + 2 * step + i, device="cuda") for i in (0, 1))
        o, lse = focus.attn_decode(cache, q, kn, vn, workspace=ws)
        focus.kv_compact_window(cache)
        qb, kb, vb = bits(q), bits(kn), bits(vn)
        o_ref, lse_ref = np.zeros((B, Hq, d)), np.zeros((B, Hq))
        for b in range(B):
            e = np.arange(Hq) // g            # K/V head of each query head
            o_ref[b], lse_ref[b] = fo.decode(qb[b], kb[b][e], vb[b][e], rk[b][e], rv[b][e], [R[b]] * Hq,
                                             wk[b][e], wv[b][e], [fill[b]] * Hq, scale)
            wk[b, :, fill[b]], wv[b, :, fill[b]] = kb[b], vb[b]
            fill[b] += 1
            kw = int(k_sched[widx[b]])
            if fill[b] == W + -(-W // kw):
                keep_rows = fo.window_retained_rows(W, kw, True, 0)
                rk[b, :, R[b]:R[b] + keep_rows.size] = wk[b][:, keep_rows]
                rv[b, :, R[b]:R[b] + keep_rows.size] = wv[b][:, keep_rows]
                R[b] += keep_rows.size
                fill[b] = 0
                widx[b] += 1
        assert_attn_close(o, lse, o_ref, lse_ref, f"gqa decode g={g} step {step}")
    torch.cuda.synchronize()
    assert np.array_equal(cache.ring_len.cpu().numpy(), R)
    assert np.array_equal(cache.win_fill.cpu().numpy(), fill)


def test_gqa_rejects_mismatched_heads():
    cache = focus.Cache(1, 2, 64, C_ring=16, q_per_kv=4)
    L = focus.layout(100, 100, [10])
    q = torch.zeros((1, 2, L["T"], 64), dtype=torch.bfloat16, device="cuda")   # needs 8 query heads
    with pytest.raises(ValueError):
        focus.attn_prefill(cache, q, q, q, L)


@pytest.mark.parametrize("g,d", [(2, 64), (8, 128), (16, 64), (16, 128)])
def test_gqa_decode_multi_split_matches_oracle(g, d):
    """Several 1,024-key splits per head with ragged tails: ring lengths 2,900 and
    1,025 (one key into the second split), window fills 3 and 0. Each query head
    group is served per K/V pass (g = 16 as two slices of eight)."""
    B, H, W, kw = 2, 2, 50, 10
    cache = focus.Cache(B, H, d, C_ring=3_000, C_win=64, W=W, k_sched=np.full(400, kw, np.int32), q_per_kv=g)
    gen = torch.Generator(device="cuda").manual_seed(23)
    for t in (cache.ring_k, cache.ring_v, cache.win_k, cache.win_v):
        t.copy_(torch.randn(t.shape, generator=gen, device="cuda").bfloat16())
    R, fill = np.array([2_900, 1_025], np.int32), np.array([3, 0], np.int32)
    cache.ring_len.copy_(torch.from_numpy(R))
    cache.win_idx.copy_(torch.tensor([7, 3], dtype=torch.int32))
    cache.win_fill.copy_(torch.from_numpy(fill))
    rk, rv, wk, wv = (bits(t).copy() for t in (cache.ring_k, cache.ring_v, cache.win_k, cache.win_v))
    Hq = H * g
    q = inputs.normal_bf16((B, Hq, d), 1.0, seed=41, device="cuda")
    kn, vn = (inputs.normal_bf16((B, H, d), 1.0, seed=s, device="cuda") for s in (42, 43))
    o, lse = focus.attn_decode(cache, q, kn, vn)
    qb, kb, vb = bits(q), bits(kn), bits(vn)
    o_ref, lse_ref = np.zeros((B, Hq, d)), np.zeros((B, Hq))
    e = np.arange(Hq) // g
    for b in range(B):
        o_ref[b], lse_ref[b] = fo.decode(qb[b], kb[b][e], vb[b][e], rk[b][e], rv[b][e], [R[b]] * Hq,
                                         wk[b][e], wv[b][e], [fill[b]] * Hq, 1 / math.sqrt(d))
    assert_attn_close(o, lse, o_ref, lse_ref, f"gqa decode multi-split g={g} d={d}")
    assert np.array_equal(cache.win_fill.cpu().numpy(), fill + 1)
