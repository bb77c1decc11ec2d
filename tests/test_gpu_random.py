"""Seeded randomized sweep of the prefill path against the fp64 oracle: each case
draws its own head dimension, batch, K/V heads and grouped-query factor, sequence
length, fixed or adaptive windows, per-window cadences (including k = 0, k = 1 and
k > W), boundary tail, mask (App. A's appendix mask or Sec. 3.2's k-mer-local
mask), rotary embedding and ring capacity (which selects the persistent or the
one-CTA-per-item kernel). The layout must match bit for bit and every output row
must meet the parity tolerance. A second sweep draws random decode caches
(per-sequence ring lengths, fills and window indices, W, cadences, tails, grouped
heads) and checks 40 decode steps each. FOCUS_RANDOM_PREFILL_SEEDS and
FOCUS_RANDOM_DECODE_SEEDS widen the sweeps (the same generators, more seeds)."""
import math
import os

import numpy as np
import pytest
import torch

from oracle import focus_oracle as fo
from paper_2511_14694_gb300 import focus, inputs, pipeline
from test_gpu_parity import PER_ITEM_C_RING, assert_attn_close

pytestmark = pytest.mark.gpu

K_CHOICES = [0, 1, 2, 3, 7, 10, 50, 100, 5_000]
N_PREFILL = int(os.environ.get("FOCUS_RANDOM_PREFILL_SEEDS", "128"))
N_DECODE = int(os.environ.get("FOCUS_RANDOM_DECODE_SEEDS", "48"))


@pytest.fixture(autouse=True)
def _clean_status():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    focus.device_status(clear=True)
    yield
    assert focus.device_status(clear=True) == 0, "a kernel reported an error"


def _draw(seed):
    r = np.random.default_rng(seed)
    case = dict(d=int(r.choice([64, 128])), B=int(r.integers(1, 3)), H=int(r.integers(1, 4)),
                g=int(r.choice([1, 1, 2, 4])), N=int(r.integers(50, 3_000)),
                local=bool(r.random() < 0.35), rope=float(r.choice([0.0, 0.0, 10_000.0])),
                per_item=bool(r.random() < 0.4))
    case["tail"] = 0 if case["local"] else int(r.choice([0, 0, 3]))
    if r.random() < 0.5:
        case["W"] = int(r.integers(16, 1_500))
        M = -(-case["N"] // case["W"])
    else:                                       # adaptive window lengths (Sec. 5)
        lens = r.integers(8, 1_200, size=4 * case["N"] // 8 + 4).astype(np.int32)
        case["W"] = fo.window_schedule(case["N"], lens)
        M = case["W"].size
    ks = np.asarray(r.choice(K_CHOICES, size=M), np.int32)
    if (ks == 1).any() and case["N"] > 1_500:   # every base followed by a summary: keep the oracle quick
        ks[ks == 1] = 2
    case["k"] = ks
    return case


@pytest.mark.parametrize("seed", range(N_PREFILL))
def test_random_prefill_matches_oracle(seed):
    c = _draw(seed)
    d, B, H, g, N, W, k, tail = c["d"], c["B"], c["H"], c["g"], c["N"], c["W"], c["k"], c["tail"]
    L = focus.layout(N, W, k, tail=tail)
    ref = fo.layout(N, W, k, tail=tail)
    for name in ("kind", "pos", "win", "keep", "win_off", "ring_off"):
        assert np.array_equal(L[name].cpu().numpy(), ref[name]), (c, name)
    assert np.array_equal(L["sum_idx"].cpu().numpy(), ref["sum_idx"]), c
    T, Hq = L["T"], H * g
    q = inputs.normal_bf16((B, Hq, T, d), 1.0, seed=1_000 + seed, device="cuda")
    kk, v = (inputs.normal_bf16((B, H, T, d), 1.0, seed=2_000 + 2 * seed + i, device="cuda") for i in (0, 1))
    cache = focus.Cache(B, H, d, C_ring=PER_ITEM_C_RING if c["per_item"] else max(L["R"], 1), k_sched=k,
                        tail=tail, q_per_kv=g, rope_theta=c["rope"])
    flags = focus.PREFILL_KMER_LOCAL if c["local"] else 0
    o, lse = pipeline.prefill_masked_parallel(cache, q, kk, v, L, flags=flags)
    torch.cuda.synchronize()
    # the oracle sees every query head with its K/V head's rows
    e = np.arange(Hq) // g
    flat = lambda t: t.cpu().reshape(B * t.shape[1], T, d)  # noqa: E731
    qh = flat(q)
    kh, vh = flat(kk[:, e]), flat(v[:, e])
    heads, rows = np.repeat(np.arange(B * Hq), T), np.tile(np.arange(T), B * Hq)
    scale = 1 / math.sqrt(d)
    if c["rope"]:
        pos = np.arange(T)
        qr, kr = fo.rope(qh, pos, c["rope"], round_bf16=True), fo.rope(kh, pos, c["rope"], round_bf16=True)
    if c["local"]:
        if c["rope"]:     # rotated rows rounded to bf16 are exact bf16 inputs
            qh, kh = (torch.from_numpy(x.astype(np.float32)).bfloat16() for x in (qr, kr))
        o_ref, lse_ref = fo.attn_rows_kmer_local(qh, kh, vh, ref["kind"], ref["win"], fo.layout_kmer(N, W, k),
                                                 scale, heads, rows)
    elif c["rope"]:
        o_ref, lse_ref = fo.attn_rows_f64(qr, kr, vh, ref["keep"], ref["win"], scale, heads, rows)
    else:
        o_ref, lse_ref = fo.attn_rows(qh, kh, vh, ref["keep"], ref["win"], scale, heads, rows)
    assert_attn_close(o, lse, o_ref.reshape(B, Hq, T, d), lse_ref.reshape(B, Hq, T), str(c))


@pytest.mark.parametrize("seed", range(N_DECODE))
def test_random_decode_matches_oracle(seed):
    """Decode steps (App. A.2) on random caches: per-sequence ring lengths, window
    fills, window indices and (with the rotary embedding) first positions, window
    length W, cadences (k = 0: no summary rows), boundary tails and grouped heads;
    40 steps against the oracle with the cache evolved on the host (the window's
    kept rows join the ring when it is full)."""
    r = np.random.default_rng(10_000 + seed)
    d, B, H = int(r.choice([64, 128])), int(r.integers(1, 5)), int(r.integers(1, 4))
    g, W, tail = int(r.choice([1, 2, 3, 4, 8])), int(r.integers(8, 100)), int(r.choice([0, 0, 2]))
    k_sched = np.asarray(r.choice([0, 1, 2, 3, 5, 10, W, W + 7], size=64), np.int32)
    theta = float(r.choice([0.0, 0.0, 10_000.0, 500_000.0]))
    Tws = np.array([W + (-(-W // kk) if kk > 0 else 0) for kk in k_sched])
    widx = r.integers(0, 8, size=B).astype(np.int32)
    fill = np.array([r.integers(0, Tws[w]) for w in widx], np.int32)
    R = r.integers(0, 300, size=B).astype(np.int32)
    cache = focus.Cache(B, H, d, C_ring=int(R.max()) + 2 * W + 128, C_win=int(Tws.max()) + 8, W=W, k_sched=k_sched,
                        tail=tail, q_per_kv=g, rope_theta=theta)
    gen = torch.Generator(device="cuda").manual_seed(seed)
    for t in (cache.ring_k, cache.ring_v, cache.win_k, cache.win_v):
        t.copy_(torch.randn(t.shape, generator=gen, device="cuda").bfloat16())
    cache.ring_len.copy_(torch.from_numpy(R))
    cache.win_idx.copy_(torch.from_numpy(widx))
    cache.win_fill.copy_(torch.from_numpy(fill))
    if theta:
        cache.pos_base.copy_(torch.from_numpy(r.integers(0, 1_000_000, size=B).astype(np.int32)))
        _rope_decode_steps(cache, W, k_sched, theta, tail, g, seed)
        return
    bits_ = lambda t: t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)  # noqa: E731
    rk, rv, wk, wv = (bits_(t).copy() for t in (cache.ring_k, cache.ring_v, cache.win_k, cache.win_v))
    Rm, fm, wm = R.astype(np.int64), fill.astype(np.int64), widx.astype(np.int64)
    ws = cache.new_workspace()
    e = np.arange(H * g) // g                      # K/V head of each query head
    scale = 1 / math.sqrt(d)
    for step in range(40):
        q = inputs.normal_bf16((B, H * g, d), 1.0, seed=20_000 + 97 * seed + step, device="cuda")
        kn, vn = (inputs.normal_bf16((B, H, d), 1.0, seed=30_000 + 97 * seed + 2 * step + i, device="cuda")
                  for i in (0, 1))
        o, lse = focus.attn_decode(cache, q, kn, vn, workspace=ws)
        focus.kv_compact_window(cache)
        qb, kb, vb = bits_(q), bits_(kn), bits_(vn)
        o_ref, lse_ref = np.zeros((B, H * g, d)), np.zeros((B, H * g))
        for b in range(B):
            o_ref[b], lse_ref[b] = fo.decode(qb[b], kb[b][e], vb[b][e], rk[b][e], rv[b][e], [Rm[b]] * (H * g),
                                             wk[b][e], wv[b][e], [fm[b]] * (H * g), scale)
            wk[b, :, fm[b]], wv[b, :, fm[b]] = kb[b], vb[b]
            fm[b] += 1
            kw = int(k_sched[wm[b]])
            if fm[b] == Tws[wm[b]]:                # window complete: its kept rows join the ring
                keep = fo.window_retained_rows(W, kw, True, tail)
                rk[b, :, Rm[b]:Rm[b] + keep.size] = wk[b][:, keep]
                rv[b, :, Rm[b]:Rm[b] + keep.size] = wv[b][:, keep]
                Rm[b] += keep.size
                fm[b] = 0
                wm[b] += 1
        assert_attn_close(o, lse, o_ref, lse_ref, f"seed {seed} step {step}: d={d} B={B} H={H} g={g} W={W} tail={tail}")
    torch.cuda.synchronize()
    assert np.array_equal(cache.ring_len.cpu().numpy(), Rm)
    assert np.array_equal(cache.win_fill.cpu().numpy(), fm)


def _rope_decode_steps(cache, W, k_sched, theta, tail, g, seed):
    """The rotary case of the sweep: q and k_new rotated at pos_base + fill, the
    host mirror of test_gpu_rope.py evolving the rotated keys."""
    from test_gpu_rope import RopeDecodeModel
    B, H, d = cache.B, cache.H, cache.d
    model = RopeDecodeModel(cache, W, k_sched, theta, tail)
    ws = cache.new_workspace()
    scale = 1 / math.sqrt(d)
    for step in range(40):
        q = inputs.normal_bf16((B, H * g, d), 1.0, seed=20_000 + 97 * seed + step, device="cuda")
        kn, vn = (inputs.normal_bf16((B, H, d), 1.0, seed=30_000 + 97 * seed + 2 * step + i, device="cuda")
                  for i in (0, 1))
        o, lse = focus.attn_decode(cache, q, kn, vn, workspace=ws)
        focus.kv_compact_window(cache)
        o_ref, lse_ref = model.step(q, kn, vn, scale)
        assert_attn_close(o, lse, o_ref, lse_ref, f"seed {seed} step {step}: rope {theta} d={d} B={B} H={H} g={g} "
                                                  f"W={W} tail={tail}")
    torch.cuda.synchronize()
    assert np.array_equal(cache.ring_len.cpu().numpy(), model.R)
    assert np.array_equal(cache.win_fill.cpu().numpy(), model.fill)
    assert np.array_equal(cache.pos_base.cpu().numpy(), model.pos)
