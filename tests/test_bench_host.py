"""CPU checks of the host arithmetic behind the bench line: the visible-pair and
k-mer-local key counts that set the algorithmic FLOPs and bytes of a roofline,
the oracle baseline's whole-workload time, the weak-scaling value and the
roofline fraction. Each count is compared with the oracle's own visibility (the
brute-force predicate, or ln |visible| from attention over zero scores)."""
import math

import numpy as np
import pytest
import torch

import bench
from oracle import focus_oracle as fo
from paper_2511_14694_gb300 import inputs

CASES = [
    # N, W, k schedule (cycled), boundary tail
    (700, 60, [1, 7, 13, 0, 60, 100], 0),
    (1_000, 100, [10], 0),
    (997, 128, [3, 200, 17], 2),
    (64, 1_000, [0], 0),                     # one window, no summaries: plain causal
]


def _k(N, W, ks):
    M = -(-N // W)
    return np.resize(np.asarray(ks, np.int32), M)


@pytest.mark.parametrize("N,W,ks,tail", CASES)
def test_visible_pairs_equals_the_brute_force_predicate(N, W, ks, tail):
    """Appendix visibility: j <= i and (same window or j retained)."""
    k = _k(N, W, ks)
    L = fo.layout(N, W, k, tail=tail)
    win, keep = L["win"].astype(np.int64), L["keep"].astype(bool)
    T = L["T"]
    i, j = np.tril_indices(T)
    brute = int(((win[i] == win[j]) | keep[j]).sum())
    assert bench.visible_pairs(L["win_off"], L["ring_off"]) == brute


@pytest.mark.parametrize("N,W,ks,tail", [c for c in CASES if c[3] == 0])
def test_kmer_local_row_counts_equal_the_oracle_visibility(N, W, ks, tail):
    """q = 0 gives LSE_i = ln |visible(i)| under the oracle's k-mer-local rule."""
    k = _k(N, W, ks)
    L = fo.layout(N, W, k)
    T = L["T"]
    q = torch.zeros((1, T, 8), dtype=torch.bfloat16)
    _, kk, v = inputs.qkv((1, T, 8), seed=3)
    _, lse = fo.attn_rows_kmer_local(q, kk, v, L["kind"], L["win"], fo.layout_kmer(N, W, k), 1.0,
                                     np.zeros(T, np.int64), np.arange(T))
    counts = bench.kmer_local_row_counts(L["win_off"], L["ring_off"], k)
    np.testing.assert_allclose(np.log(counts), lse, rtol=0, atol=1e-12)


def test_oracle_baseline_in_full_and_extrapolated():
    cfg = dict(B=2, H=4, N=1_000)
    secs_full = [1.0, 2.0, 3.0, 4.0, 5.0, 6.0, 7.0, 8.0]        # all B x H passes ran
    val, desc, full_s = bench.oracle_baseline(cfg, secs_full, "appendix")
    assert full_s == pytest.approx(36.0) and val == pytest.approx(2 * 1_000 / 36.0)
    assert "timed in full" in desc
    val, desc, full_s = bench.oracle_baseline(cfg, [1.0, 3.0, 2.0], "appendix")   # a sample
    assert full_s == pytest.approx(8 * 2.0) and val == pytest.approx(2 * 1_000 / 16.0)
    assert "extrapolated" in desc


def test_weak_scaling_value_counts_every_rank():
    assert bench.weak_scaling_value(1_000.0, 4, 2.0) == pytest.approx(2_000.0)


def test_prefill_roofline_fraction_and_labels():
    peaks = {"bf16_tflops": 2_000.0, "bf16_tflops_sustained": 1_600.0, "hbm_gbs": 8_000.0}
    pre = dict(attn_launches_per_step=1, flops_per_step=2.0e12, attn_ms=2.0, pairs=10, kernel="tcgen05 persistent",
               local_mask=False, bytes_per_step=4.0e9)
    r = bench.prefill_roofline(pre, peaks, "measured")
    assert r["achieved"] == pytest.approx(1_000.0) and r["frac"] == pytest.approx(0.5)
    assert r["frac_of_sustained"] == pytest.approx(0.625) and r["unit"] == "TFLOP/s"
    pre["kernel"] = "rotation pass + tcgen05 persistent"
    assert "rotation pass" in bench.prefill_roofline(pre, peaks, "measured")["kernel"]
    pre.update(local_mask=True, kernel="tcgen05 k-mer tiles")
    r = bench.prefill_roofline(pre, peaks, "measured")
    assert r["bound"] == "hbm" and r["achieved"] == pytest.approx(2_000.0) and r["frac"] == pytest.approx(0.25)
    assert math.isfinite(r["tflops"])
