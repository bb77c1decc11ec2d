"""GPU parity of the rotary position embedding (RoFormer rotation at the
layout's position ids) against the fp64 oracle: masked-parallel and streaming
prefill, the rotated ring written by bulk compaction, decode with window
roll-over, and a 1 Mb stream whose positions reach ~10^6.

The rotated rows of a bf16 path are bf16: the oracle rotates in fp64 and rounds
once to bf16 (nearest, ties to even); the kernels rotate in fp32 and round once,
so the two can differ by one bf16 step where the exact value lies near a
rounding boundary. Attention uses the bars of test_gpu_parity; stored rotated
keys are compared within half a bf16 step (2^-8 relative) of the exact rotation,
or within one step (2^-7) of the oracle's rounded rows.
"""
import math

import numpy as np
import pytest
import torch

from oracle import focus_oracle as fo
from paper_2511_14694_gb300 import focus, inputs, pipeline
from test_gpu_parity import assert_attn_close, bits

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _clean_status():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    focus.device_status(clear=True)
    yield
    assert focus.device_status(clear=True) == 0, "a kernel reported an error"


def assert_keys_close(gpu_bf16, ref_f64, what="", rel=2.0 ** -8):
    """rel = 2^-8: one rounding of the exact value; 2^-7: against a reference that
    was itself rounded (the two may pick neighbouring bf16 values)."""
    g = gpu_bf16.detach().float().cpu().double().numpy()
    err = np.abs(g - ref_f64)
    bound = rel * np.abs(ref_f64) + 1e-5
    assert (err <= bound).all(), f"{what}: worst excess {(err - bound).max():.3e}"


def _case(N, W, ks, B, H, d, theta, seed, std=1.0):
    M = -(-N // W)
    k = np.resize(np.asarray(ks, np.int32), M)
    L = focus.layout(N, W, k)
    q, kk, v = inputs.qkv((B, H, L["T"], d), std=std, seed=seed, device="cuda")
    cache = focus.Cache(B, H, d, C_ring=max(L["R"], 1), k_sched=k, rope_theta=theta)
    return L, k, q, kk, v, cache


def _ref_all_rows(N, W, k, q, kk, v, theta):
    B, H, T, d = q.shape
    ref_L = fo.layout(N, W, k)
    pos = np.arange(T)
    qf = fo.rope(q.reshape(B * H, T, d).cpu(), pos, theta, round_bf16=True)
    kf = fo.rope(kk.reshape(B * H, T, d).cpu(), pos, theta, round_bf16=True)
    heads, rows = np.repeat(np.arange(B * H), T), np.tile(np.arange(T), B * H)
    o, lse = fo.attn_rows_f64(qf, kf, v.reshape(B * H, T, d).cpu(), ref_L["keep"], ref_L["win"],
                              1.0 / math.sqrt(d), heads, rows)
    return o.reshape(B, H, T, d), lse.reshape(B, H, T), kf.reshape(B, H, T, d), ref_L


ROPE_CASES = [
    # N, W, k schedule (cycled), B, H, d, rope base
    (4_000, 1_000, [100], 1, 2, 64, 10_000.0),
    (5_000, 1_024, [100], 1, 2, 128, 500_000.0),
    (3_001, 300, [1, 7, 50, 0, 300, 1_000], 2, 1, 128, 10_000.0),
    (300, 64, [64], 1, 2, 64, 1_000.0),
]


# with the workspace a pass rotates q and k once before the attention; without it
# the one-CTA-per-item kernel rotates each tile it loads
@pytest.mark.parametrize("ws,kernel", [("auto", "rotation pass + tcgen05 persistent"),
                                       (None, "tcgen05, one CTA per work item")])
@pytest.mark.parametrize("N,W,ks,B,H,d,theta", ROPE_CASES)
def test_prefill_rope_masked_parallel_matches_oracle(N, W, ks, B, H, d, theta, ws, kernel):
    L, k, q, kk, v, cache = _case(N, W, ks, B, H, d, theta, seed=N + 3)
    assert focus.prefill_kernel(cache, q, kk, v, L, workspace=ws) == kernel
    o, lse = pipeline.prefill_masked_parallel(cache, q, kk, v, L, workspace=ws)
    torch.cuda.synchronize()
    o_ref, lse_ref, kf, ref_L = _ref_all_rows(N, W, k, q, kk, v, theta)
    assert_attn_close(o, lse, o_ref, lse_ref, f"rope N={N} W={W} k={ks}")
    # the ring holds the FOCUS rows' keys rotated at their position ids, values as they were
    R = L["R"]
    assert_keys_close(cache.ring_k[:, :, :R], kf[:, :, ref_L["sum_idx"]], "ring K", rel=2.0 ** -7)
    assert np.array_equal(bits(cache.ring_v)[:, :, :R], bits(v)[:, :, ref_L["sum_idx"]])


@pytest.mark.parametrize("ws", ["auto", None])
@pytest.mark.parametrize("g,d", [(4, 128), (3, 64)])
def test_prefill_rope_grouped_heads_match_oracle(g, d, ws):
    """Grouped-query heads with the rotary embedding: query head hq uses K/V head
    hq // g; every query head and K/V head is rotated at the layout's positions."""
    N, W, ks, B, Hk, theta = 3_000, 1_000, [100, 50, 7], 2, 2, 10_000.0
    M = -(-N // W)
    k = np.resize(np.asarray(ks, np.int32), M)
    L = focus.layout(N, W, k)
    q = inputs.normal_bf16((B, Hk * g, L["T"], d), 1.0, seed=81, device="cuda")
    kk = inputs.normal_bf16((B, Hk, L["T"], d), 1.0, seed=82, device="cuda")
    v = inputs.normal_bf16((B, Hk, L["T"], d), 1.0, seed=83, device="cuda")
    cache = focus.Cache(B, Hk, d, C_ring=L["R"], k_sched=k, rope_theta=theta, q_per_kv=g)
    o, lse = pipeline.prefill_masked_parallel(cache, q, kk, v, L, workspace=ws)
    torch.cuda.synchronize()
    T = L["T"]
    ref_L = fo.layout(N, W, k)
    pos = np.arange(T)
    qf = fo.rope(q.reshape(B * Hk * g, T, d).cpu(), pos, theta, round_bf16=True)
    kf = fo.rope(kk.reshape(B * Hk, T, d).cpu(), pos, theta, round_bf16=True)
    kv_of = np.arange(B * Hk * g) // g                  # K/V head of each (sequence, query head)
    kf_q = kf[kv_of]
    v_q = v.reshape(B * Hk, T, d).cpu()[torch.from_numpy(kv_of)]
    rows = np.arange(0, T, 3)
    heads = np.repeat(np.arange(B * Hk * g), rows.size)
    o_ref, lse_ref = fo.attn_rows_f64(qf, kf_q, v_q, ref_L["keep"], ref_L["win"], 1.0 / math.sqrt(d), heads,
                                      np.tile(rows, B * Hk * g))
    assert_attn_close(o.reshape(B * Hk * g, T, d)[:, rows], lse.reshape(B * Hk * g, T)[:, rows],
                      o_ref.reshape(B * Hk * g, rows.size, d), lse_ref.reshape(B * Hk * g, rows.size),
                      f"rope gqa g={g} ws={ws}")


@pytest.mark.parametrize("d", [64, 128])
def test_prefill_rope_streaming_matches_oracle(d):
    N, W, ks, B, H, theta = 3_000, 500, [10, 50, 0, 7, 100, 500], 2, 2, 10_000.0
    L, k, q, kk, v, cache = _case(N, W, ks, B, H, d, theta, seed=41)
    o = torch.empty_like(q)
    lse = torch.empty((B, H, L["T"]), dtype=torch.float32, device="cuda")
    off = L["win_off_host"]
    for w in range(L["M"]):
        a, e = int(off[w]), int(off[w + 1])
        sl = lambda t: t[:, :, a:e].contiguous()  # noqa: E731
        ow, lw = pipeline.prefill_window(cache, sl(q), sl(kk), sl(v), L, w)
        o[:, :, a:e] = ow
        lse[:, :, a:e] = lw
    torch.cuda.synchronize()
    o_ref, lse_ref, kf, ref_L = _ref_all_rows(N, W, k, q, kk, v, theta)
    assert_attn_close(o, lse, o_ref, lse_ref, "rope streaming")
    assert_keys_close(cache.ring_k[:, :, :L["R"]], kf[:, :, ref_L["sum_idx"]], "ring K", rel=2.0 ** -7)


class RopeDecodeModel:
    """Host mirror of the decode cache with fp64 (rotated) keys, evolved with the
    oracle's rules (App. A.2): each step rotates q and k_new at the new row's
    position id pos_base + fill, appends, and retires full windows (their summary
    rows and the last `tail` ordinary rows join the ring)."""

    def __init__(self, cache, W, k_sched, theta, tail=0):
        B, H = cache.B, cache.H
        self.g = max(cache.q_per_kv, 1)          # query heads per K/V head
        self.rk = cache.ring_k.float().cpu().double().numpy().copy()
        self.rv = bits(cache.ring_v).copy()
        self.wk = cache.win_k.float().cpu().double().numpy().copy()
        self.wv = bits(cache.win_v).copy()
        self.R = cache.ring_len.cpu().numpy().copy()
        self.fill = cache.win_fill.cpu().numpy().copy()
        self.widx = cache.win_idx.cpu().numpy().copy()
        self.pos = cache.pos_base.cpu().numpy().astype(np.int64).copy()
        self.W, self.k, self.theta, self.H, self.tail = W, np.asarray(k_sched), theta, H, tail

    def step(self, q, kn, vn, scale):
        B, Hq, d = q.shape
        e = np.arange(Hq) // self.g              # K/V head of each query head
        o, lse = np.zeros((B, Hq, d)), np.zeros((B, Hq))
        for b in range(B):
            p = self.pos[b] + self.fill[b]
            qf = fo.rope(q[b].cpu(), p, self.theta, round_bf16=True)
            kf = fo.rope(kn[b].cpu(), p, self.theta, round_bf16=True)
            o[b], lse[b] = fo.decode_f64(qf, kf[e], bits(vn[b])[e], self.rk[b][e], self.rv[b][e], [self.R[b]] * Hq,
                                         self.wk[b][e], self.wv[b][e], [self.fill[b]] * Hq, scale)
            f = self.fill[b]
            self.wk[b, :, f], self.wv[b, :, f] = kf, bits(vn[b])
            self.fill[b] += 1
            kw = int(self.k[self.widx[b]])
            Tw = self.W + (-(-self.W // kw) if kw > 0 else 0)
            if self.fill[b] == Tw:
                rows = fo.window_retained_rows(self.W, kw, True, self.tail)
                r = self.R[b]
                self.rk[b, :, r:r + rows.size] = self.wk[b][:, rows]
                self.rv[b, :, r:r + rows.size] = self.wv[b][:, rows]
                self.R[b] += rows.size
                self.fill[b] = 0
                self.widx[b] += 1
                self.pos[b] += Tw
        return o, lse


@pytest.mark.parametrize("d", [64, 128])
def test_decode_rope_steps_match_oracle(d):
    B, H, W, theta = 3, 2, 50, 10_000.0
    k_sched = np.array([10, 7, 25, 50, 3, 10, 10, 10], np.int32)
    cache = focus.Cache(B, H, d, C_ring=512, C_win=72, W=W, k_sched=k_sched, rope_theta=theta)
    g = torch.Generator(device="cuda").manual_seed(5)
    for t in (cache.ring_k, cache.ring_v, cache.win_k, cache.win_v):
        t.copy_(torch.randn(t.shape, generator=g, device="cuda").bfloat16())
    cache.ring_len.copy_(torch.tensor([0, 37, 300], dtype=torch.int32))
    cache.win_idx.copy_(torch.tensor([0, 1, 2], dtype=torch.int32))
    cache.win_fill.copy_(torch.tensor([0, 50, 20], dtype=torch.int32))   # window 1 has T_w = 58
    cache.pos_base.copy_(torch.tensor([0, 1_234, 987_000], dtype=torch.int32))
    model = RopeDecodeModel(cache, W, k_sched, theta)
    ws = cache.new_workspace()
    scale = 1.0 / math.sqrt(d)
    for step in range(70):
        q, kn, vn = inputs.qkv((B, H, d), seed=300 + step, device="cuda")
        o, lse = focus.attn_decode(cache, q, kn, vn, workspace=ws)
        focus.kv_compact_window(cache)
        o_ref, lse_ref = model.step(q, kn, vn, scale)
        assert_attn_close(o, lse, o_ref, lse_ref, f"rope decode step {step}")
    torch.cuda.synchronize()
    assert np.array_equal(cache.ring_len.cpu().numpy(), model.R)
    assert np.array_equal(cache.win_fill.cpu().numpy(), model.fill)
    assert np.array_equal(cache.pos_base.cpu().numpy(), model.pos)
    for b in range(B):
        R, f = int(model.R[b]), int(model.fill[b])
        assert_keys_close(cache.ring_k[b, :, :R], model.rk[b, :, :R], f"ring K b={b}", rel=2.0 ** -7)
        assert_keys_close(cache.win_k[b, :, :f], model.wk[b, :, :f], f"window K b={b}", rel=2.0 ** -7)


@pytest.mark.parametrize("g,d", [(4, 128), (3, 64), (8, 64)])
def test_decode_rope_grouped_heads_match_oracle(g, d):
    """The rotary embedding with grouped-query heads: q rotated per query head,
    k_new per K/V head, on the tensor-core kernel (even g) and the CUDA-core one
    (odd g), across window retirements."""
    B, H, W, theta = 2, 2, 50, 10_000.0
    k_sched = np.array([10, 25, 7, 50, 10, 10], np.int32)
    cache = focus.Cache(B, H, d, C_ring=256, C_win=64, W=W, k_sched=k_sched, rope_theta=theta, q_per_kv=g)
    gen = torch.Generator(device="cuda").manual_seed(17)
    for t in (cache.ring_k, cache.ring_v, cache.win_k, cache.win_v):
        t.copy_(torch.randn(t.shape, generator=gen, device="cuda").bfloat16())
    cache.ring_len.copy_(torch.tensor([20, 130], dtype=torch.int32))
    cache.win_idx.copy_(torch.tensor([1, 2], dtype=torch.int32))
    cache.win_fill.copy_(torch.tensor([40, 3], dtype=torch.int32))
    cache.pos_base.copy_(torch.tensor([5_000, 77_777], dtype=torch.int32))
    model = RopeDecodeModel(cache, W, k_sched, theta)
    ws = cache.new_workspace()
    scale = 1.0 / math.sqrt(d)
    for step in range(30):
        q = inputs.normal_bf16((B, H * g, d), 1.0, seed=500 + step, device="cuda")
        kn, vn = (inputs.normal_bf16((B, H, d), 1.0, seed=800 + 2 * step + i, device="cuda") for i in (0, 1))
        o, lse = focus.attn_decode(cache, q, kn, vn, workspace=ws)
        focus.kv_compact_window(cache)
        o_ref, lse_ref = model.step(q, kn, vn, scale)
        assert_attn_close(o, lse, o_ref, lse_ref, f"rope gqa g={g} decode step {step}")
    torch.cuda.synchronize()
    assert np.array_equal(cache.ring_len.cpu().numpy(), model.R)
    assert np.array_equal(cache.pos_base.cpu().numpy(), model.pos)


def test_full_size_streaming_rope_sampled():
    """Batch 4, N = 1 Mb, W = 1,000, k = 100, 32 heads, d = 128, base 500,000: one
    prefill and one compaction per window; positions reach 1,009,999. Sampled
    windows of two heads against the oracle, which sees each row's visible set
    (the ring rows before its window, then its window up to itself) rotated at
    the rows' true position ids."""
    from paper_2511_14694_gb300.workloads import WORKLOADS
    cfg = WORKLOADS["stream_1mb_b4_h32_d128"]
    B, N, W, H, d, P = cfg["B"], cfg["N"], cfg["W"], cfg["H"], cfg["d"], cfg["pool"]
    theta = 500_000.0
    M = -(-N // W)
    L = focus.layout(N, W, [cfg["k"][0]])
    off, roff = L["win_off_host"], L["ring_off_host"]
    Tw = int(off[1] - off[0])
    pq, pk, pv = inputs.qkv((P, B, H, Tw, d), std=cfg["std"], seed=inputs.DEFAULT_SEED, device="cuda")
    cache = focus.Cache(B, H, d, C_ring=L["R"], rope_theta=theta)
    want = [0, 1, 998, 999]
    b, heads = 1, [0, 17]
    got = {}
    for w in range(M):
        o, lse = pipeline.prefill_window(cache, pq[w % P], pk[w % P], pv[w % P], L, w)
        if w in want:
            got[w] = (o[b, heads].cpu(), lse[b, heads].cpu())
    torch.cuda.synchronize()
    ref_L = fo.layout(N, W, [cfg["k"][0]])
    sum_idx = ref_L["sum_idx"]
    for i, h in enumerate(heads):
        pq_h, pk_h, pv_h = (t[:, b, h].cpu() for t in (pq, pk, pv))     # [P, T_w, d]
        for w in want:
            a, e = int(off[w]), int(off[w + 1])
            R_w = int(roff[w])
            ring_rows = sum_idx[:R_w]                         # augmented indices of the retained rows
            src_w = torch.from_numpy(ring_rows // Tw)         # every window has T_w rows here
            in_w = torch.from_numpy(ring_rows % Tw)
            ring_k, ring_v = pk_h[src_w % P, in_w], pv_h[src_w % P, in_w]
            kf = np.concatenate([fo.rope(ring_k, ring_rows, theta, round_bf16=True).reshape(R_w, d),
                                 fo.rope(pk_h[w % P], np.arange(a, e), theta, round_bf16=True)])
            qf = np.concatenate([np.zeros((R_w, d)), fo.rope(pq_h[w % P], np.arange(a, e), theta, round_bf16=True)])
            vv = torch.cat([ring_v, pv_h[w % P]])
            keep = np.concatenate([np.ones(R_w, np.uint8), np.zeros(e - a, np.uint8)])
            win = np.concatenate([np.zeros(R_w, np.int32), np.ones(e - a, np.int32)])
            rows = np.arange(R_w, R_w + e - a)
            o_ref, lse_ref = fo.attn_rows_f64(qf[None], kf[None], vv[None], keep, win, 1.0 / math.sqrt(d),
                                              np.zeros(rows.size, np.int64), rows)
            assert_attn_close(got[w][0][i], got[w][1][i], o_ref, lse_ref, f"rope stream w={w} h={h}")


@pytest.mark.parametrize("g,d,B,H", [(1, 128, 1, 16), (4, 64, 1, 4), (1, 64, 2, 8)])
def test_prefill_rope_kmer_tiled_matches_oracle(g, d, B, H):
    """The k-mer-local mask (Sec. 3.2) with the rotary embedding on the k-mer-tiled
    kernel (17 windows x 10 tiles x 16 query heads per sequence: above its 2,048-item
    threshold), which rotates each item's Q tile and the window rows of its K tile
    in shared memory and needs no workspace; the ring rows come rotated from the
    compaction. Every row against the oracle on the rows rotated at their positions
    and rounded to bf16, including a ragged last window."""
    N, W, k_, theta = 16_037, 1_000, 100, 500_000.0
    k = np.full(-(-N // W), k_, np.int32)
    L = focus.layout(N, W, k)
    T = L["T"]
    q = inputs.normal_bf16((B, H * g, T, d), 1.0, seed=91, device="cuda")
    kk, v = (inputs.normal_bf16((B, H, T, d), 1.0, seed=s, device="cuda") for s in (92, 93))
    cache = focus.Cache(B, H, d, C_ring=L["R"], k_sched=k, q_per_kv=g, rope_theta=theta)
    fl = focus.PREFILL_KMER_LOCAL
    assert focus.prefill_workspace_bytes(cache, q, kk, v, L, flags=fl) == 0
    assert focus.prefill_kernel(cache, q, kk, v, L, flags=fl) == "tcgen05 k-mer tiles"
    o, lse = pipeline.prefill_masked_parallel(cache, q, kk, v, L, flags=fl)
    torch.cuda.synchronize()
    ref = fo.layout(N, W, k)
    Hq = H * g
    pos = np.arange(T)
    qf = fo.rope(q.reshape(B * Hq, T, d).cpu(), pos, theta, round_bf16=True)
    kf = fo.rope(kk.reshape(B * H, T, d).cpu(), pos, theta, round_bf16=True)
    kv_of = np.arange(B * Hq) // g                      # K/V head of each (sequence, query head)
    to_bf16 = lambda x: torch.from_numpy(x.astype(np.float32)).bfloat16()  # noqa: E731 (exact: rounded rows)
    heads, rows = np.repeat(np.arange(B * Hq), T), np.tile(np.arange(T), B * Hq)
    o_ref, lse_ref = fo.attn_rows_kmer_local(to_bf16(qf), to_bf16(kf[kv_of]),
                                             v.reshape(B * H, T, d).cpu()[torch.from_numpy(kv_of)],
                                             ref["kind"], ref["win"], fo.layout_kmer(N, W, k), 1 / math.sqrt(d),
                                             heads, rows)
    assert_attn_close(o, lse, o_ref.reshape(B, Hq, T, d), lse_ref.reshape(B, Hq, T), f"rope k-mer tiles g={g} d={d}")


def test_rotation_pass_rows_match_oracle():
    """The rotation pass on its own: after a call that takes it (one query head per
    K/V head, a span of windows 2..4 so that positions start at win_off[2]), the
    workspace holds the span's q and k rows rotated at their position ids (its
    documented layout: counters, then q, then k), each within one bf16 step of the
    oracle's rotation rounded to bf16."""
    N, W, ks, B, H, d, theta = 5_000, 1_000, [100, 7, 50], 2, 2, 128, 500_000.0
    M = -(-N // W)
    k = np.resize(np.asarray(ks, np.int32), M)
    L = focus.layout(N, W, k)
    off = L["win_off_host"]
    w0, w1 = 2, 5
    a, e = int(off[w0]), int(off[w1])
    q, kk, v = inputs.qkv((B, H, e - a, d), std=1.0, seed=61, device="cuda")
    cache = focus.Cache(B, H, d, C_ring=L["R"], k_sched=k, rope_theta=theta)
    ws = focus.new_prefill_workspace(cache, q, kk, v, L, w0, w1)
    assert focus.prefill_kernel(cache, q, kk, v, L, w0, w1, workspace=ws).startswith("rotation pass + ")
    focus.attn_prefill(cache, q, kk, v, L, w0, w1, workspace=ws)
    torch.cuda.synchronize()
    T = e - a
    counters = (B * H * 4 + 255) // 256 * 256
    n = B * H * T * d * 2
    q_rot = ws[counters:counters + n].view(torch.bfloat16).reshape(B * H, T, d)
    k_rot = ws[counters + n:counters + 2 * n].view(torch.bfloat16).reshape(B * H, T, d)
    pos = a + np.arange(T)                               # the span's rows are consecutive augmented rows
    qf = fo.rope(q.reshape(B * H, T, d).cpu(), pos, theta, round_bf16=True)
    kf = fo.rope(kk.reshape(B * H, T, d).cpu(), pos, theta, round_bf16=True)
    assert_keys_close(q_rot, qf, "rotated q", rel=2.0 ** -7)
    assert_keys_close(k_rot, kf, "rotated k", rel=2.0 ** -7)
