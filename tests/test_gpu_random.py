"""Seeded randomized sweep of the prefill path against the fp64 oracle: each case
draws its own head dimension, batch, K/V heads and grouped-query factor, sequence
length, fixed or adaptive windows, per-window cadences (including k = 0, k = 1 and
k > W), boundary tail, mask (App. A's appendix mask or Sec. 3.2's k-mer-local
mask), rotary embedding and ring capacity (which selects the persistent or the
one-CTA-per-item kernel). The layout must match bit for bit and every output row
must meet the parity tolerance."""
import math

import numpy as np
import pytest
import torch

from oracle import focus_oracle as fo
from paper_2511_14694_gb300 import focus, inputs, pipeline
from test_gpu_parity import PER_ITEM_C_RING, assert_attn_close

pytestmark = pytest.mark.gpu

K_CHOICES = [0, 1, 2, 3, 7, 10, 50, 100, 5_000]


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


@pytest.mark.parametrize("seed", range(64))
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
