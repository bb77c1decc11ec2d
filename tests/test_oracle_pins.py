"""Pins the fp64 oracle to facts fixed by the paper and by mathematics, not to
itself: closed forms of the layout (App. A), a hand-spelled Fig. 1 layout, an
independent string construction, a KV-retention simulation that builds the
visible sets from the streaming process (App. A.2) instead of the visibility
predicate, exact reductions to causal attention (library SDPA), invariants
(rows of P sum to one, LSE of zero scores counts the visible set), the
sequential == masked-parallel equivalence (App. A.1) and decode == prefill.
"""
import math
import os

import numpy as np
import pytest
import scipy.special
import torch

from oracle import focus_oracle as fo
from paper_2511_14694_gb300 import inputs

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _ceil(a, b):
    return -(-a // b)


# ----------------------------------------------------------------------------- layout

LAYOUT_CASES = [
    (4_000, 1_000, [100]),
    (1_000, 1_024, [100]),          # one partial window, W mod k != 0 (Table: W=1024, k=100)
    (5_000, 1_024, [100]),
    (10, 4, [3]),                    # Fig. 1 shape
    (37, 7, [1]),
    (37, 7, [7]),
    (37, 7, [9]),                    # k > W: one summary per window
    (50, 50, [0]),                   # compression disabled
    (2_500, 1_000, [10, 25, 200]),   # per-window cadence
]


@pytest.mark.parametrize("N,W,ks", LAYOUT_CASES)
def test_layout_sizes_closed_form(N, W, ks):
    M = _ceil(N, W)
    k = inputs.k_schedule(M, ks, seed=3)
    T, R, M2 = fo.layout_size(N, W, k)
    assert M2 == M
    n_w = [min(W, N - w * W) for w in range(M)]
    B_w = [(_ceil(n, int(kk)) if kk > 0 else 0) for n, kk in zip(n_w, k)]   # B_w = ceil(|I_w|/k)
    assert R == sum(B_w)
    assert T == N + sum(B_w)                                                  # N' = N + #summaries
    # KV budget, eq. kv-budget: R_kept <= sum_w ceil(W/k_w) + W
    assert R <= sum(_ceil(W, int(kk)) if kk > 0 else 0 for kk in k) + W


@pytest.mark.parametrize("k", [1, 4, 10, 100])
def test_layout_positions_closed_form(k):
    """k | W, full windows: base i sits at i + floor(i/k); summary j at (j+1)(k+1)-1;
    after n windows the retained count is n*W/k."""
    W, n = 100, 7
    if W % k:
        pytest.skip("needs k | W")
    N = n * W
    L = fo.layout(N, W, [k])
    base_pos = L["pos"][L["kind"] == 0]
    assert np.array_equal(base_pos, np.arange(N) + np.arange(N) // k)
    assert np.array_equal(L["sum_idx"], (np.arange(N // k) + 1) * (k + 1) - 1)
    assert np.array_equal(L["ring_off"], np.arange(n + 1) * (W // k))
    assert np.array_equal(L["pos"], np.arange(L["T"]))
    assert np.array_equal(L["win_off"], np.arange(n + 1) * (W + W // k))


def _cuts(N, W):
    """Window boundaries: multiples of an integer W, or the running sums of a
    per-window schedule, up to N."""
    if np.ndim(W) == 0:
        return list(range(0, N, W)) + [N]
    cuts = [0]
    for x in W:
        if cuts[-1] >= N:
            break
        cuts.append(min(N, cuts[-1] + int(x)))
    return cuts


def _string_layout(seq, W, ks, close_tail=True):
    """Independent construction: cut the base string into windows, each window
    into k-chunks, and write 'S' after every chunk (the last chunk of the final
    window only if close_tail)."""
    out = []
    cuts = _cuts(len(seq), W)
    M = len(cuts) - 1
    for w in range(M):
        chunk = seq[cuts[w]:cuts[w + 1]]
        k = int(ks[w])
        if k == 0:
            out.append(chunk)
            continue
        pieces = [chunk[i:i + k] for i in range(0, len(chunk), k)]
        for pi, p in enumerate(pieces):
            last = pi == len(pieces) - 1
            closes = len(p) == k or w < M - 1 or close_tail
            out.append(p + ("S" if (not last or closes) else ""))
    return "".join(out)


@pytest.mark.parametrize("N,W,ks", LAYOUT_CASES)
@pytest.mark.parametrize("close_tail", [True, False])
def test_layout_matches_string_construction(N, W, ks, close_tail):
    M = _ceil(N, W)
    k = inputs.k_schedule(M, ks, seed=5)
    nt = inputs.nucleotides(2, N, seed=11).numpy()
    L = fo.layout(N, W, k, nt=nt, close_tail=close_tail)
    for b in range(2):
        seq = "".join("ACGT"[x] for x in nt[b])
        expect = _string_layout(seq, W, k, close_tail)
        got = "".join("ACGTS"[x] for x in L["tok"][b])
        assert got == expect
    assert "".join("BS"[x] for x in L["kind"]) == "".join("S" if c == "S" else "B" for c in expect)


def test_layout_fig1_golden():
    rows = []
    with open(os.path.join(GOLDEN, "fig1_layout_k3_W4.txt")) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                t, kind, src, w = line.split()
                rows.append((int(t), kind, int(src), int(w)))
    L = fo.layout(10, 4, [3])
    assert L["T"] == len(rows)
    for t, kind, src, w in rows:
        assert L["pos"][t] == t
        assert "BS"[L["kind"][t]] == kind
        assert L["src"][t] == src
        assert L["win"][t] == w
    assert list(L["win_off"]) == [0, 6, 12, 15]
    assert list(L["ring_off"]) == [0, 2, 4, 5]


def test_window_retained_rows_match_layout():
    for n, k, t in [(1000, 100, 0), (1024, 100, 0), (4, 3, 0), (7, 9, 0), (5, 1, 0), (1000, 100, 3), (7, 3, 7),
                    (10, 4, 1)]:
        L = fo.layout(n, n, [k], tail=t)
        assert np.array_equal(fo.window_retained_rows(n, k, True, t), np.nonzero(L["keep"] == 1)[0])


@pytest.mark.parametrize("N,W,ks", LAYOUT_CASES)
@pytest.mark.parametrize("tail", [1, 3, 2_000])
def test_layout_tail_counts_closed_form(N, W, ks, tail):
    """Boundary tail (App. A): each window keeps its B_w summaries plus its last
    min(tail, n_w) bases; the kept bases are the window's last base rows."""
    M = _ceil(N, W)
    k = inputs.k_schedule(M, ks, seed=3)
    L = fo.layout(N, W, k, tail=tail)
    n_w = [min(W, N - w * W) for w in range(M)]
    B_w = [(_ceil(n, int(kk)) if kk > 0 else 0) for n, kk in zip(n_w, k)]
    assert L["R"] == sum(b + min(tail, n) for b, n in zip(B_w, n_w))
    for w in range(M):
        a, e = L["win_off"][w], L["win_off"][w + 1]
        bases = [j for j in range(a, e) if L["kind"][j] == 0]
        kept_bases = [j for j in range(a, e) if L["kind"][j] == 0 and L["keep"][j] == 1]
        assert kept_bases == bases[len(bases) - min(tail, len(bases)):]
    assert np.array_equal(L["keep"][L["kind"] == 1], np.ones(int((L["kind"] == 1).sum()), np.uint8))


# ----------------------------------------------------------------------------- attention


def _rand_case(N, W, ks, H, d, seed, std=1.0, tail=0):
    M = _ceil(N, W)
    k = inputs.k_schedule(M, ks, seed=seed)
    L = fo.layout(N, W, k, tail=tail)
    q, kk, v = inputs.qkv((H, L["T"], d), std=std, seed=seed)
    return L, q, kk, v


def _visible_sets_by_streaming(L, tail=0):
    """KV-retention simulation (App. A.2): process windows in order; a row sees
    the retained set plus the current window up to itself; after the window,
    only its FOCUS rows (and its last `tail` base rows) join the retained set."""
    retained, vis = [], {}
    for w in range(L["M"]):
        a, e = L["win_off"][w], L["win_off"][w + 1]
        for i in range(a, e):
            vis[i] = list(retained) + list(range(a, i + 1))
        bases = [j for j in range(a, e) if L["kind"][j] == 0]
        tail_rows = set(bases[len(bases) - min(tail, len(bases)):]) if tail else set()
        retained += [j for j in range(a, e) if L["kind"][j] == 1 or j in tail_rows]
    return vis


def _f64(x):
    return x.to(torch.float64).numpy()


ATTN_CASES = [
    (10, 4, [3], 2, 8),       # Fig. 1 shape
    (40, 7, [2], 2, 16),
    (64, 64, [5], 1, 8),      # W >= N with summaries
    (64, 9, [1], 1, 8),       # every base summarised
    (60, 10, [20], 2, 8),     # k > W
    (63, 8, [1, 2, 3, 9], 2, 16),
]


@pytest.mark.parametrize("N,W,ks,H,d", ATTN_CASES)
@pytest.mark.parametrize("tail", [0, 2])
def test_attn_matches_streaming_simulation(N, W, ks, H, d, tail):
    L, q, k, v = _rand_case(N, W, ks, H, d, seed=N + W, tail=tail)
    T = L["T"]
    scale = 1.0 / math.sqrt(d)
    heads = np.repeat(np.arange(H), T)
    rows = np.tile(np.arange(T), H)
    o, lse = fo.attn_rows(q, k, v, L["keep"], L["win"], scale, heads, rows)
    vis = _visible_sets_by_streaming(L, tail)
    qd, kd, vd = _f64(q), _f64(k), _f64(v)
    for r, (h, i) in enumerate(zip(heads, rows)):
        j = np.array(vis[i])
        s = scale * (kd[h, j] @ qd[h, i])
        p = scipy.special.softmax(s)
        np.testing.assert_allclose(o[r], p @ vd[h, j], rtol=0, atol=1e-12)
        assert abs(lse[r] - scipy.special.logsumexp(s)) <= 1e-12 * max(1.0, abs(lse[r]))


def test_no_compression_is_plain_causal():
    """k = 0 and W >= N: exactly causal attention (App. A.2: the interface reduces
    to the base decoder), checked against torch's SDPA in fp64."""
    N, H, d = 96, 3, 32
    L, q, k, v = _rand_case(N, N, [0], H, d, seed=1)
    assert L["T"] == N and L["R"] == 0
    heads = np.repeat(np.arange(H), N)
    rows = np.tile(np.arange(N), H)
    o, lse = fo.attn_rows(q, k, v, L["keep"], L["win"], 1.0 / math.sqrt(d), heads, rows)
    qd, kd, vd = (x.to(torch.float64) for x in (q, k, v))
    ref = torch.nn.functional.scaled_dot_product_attention(qd, kd, vd, is_causal=True)
    np.testing.assert_allclose(o.reshape(H, N, d), ref.numpy(), rtol=0, atol=1e-12)
    s = (qd @ kd.transpose(-1, -2)) / math.sqrt(d)
    s = s.masked_fill(torch.triu(torch.ones(N, N, dtype=torch.bool), 1), float("-inf"))
    np.testing.assert_allclose(lse.reshape(H, N), torch.logsumexp(s, -1).numpy(), rtol=1e-13, atol=0)


def test_single_window_with_summaries_is_causal_over_augmented():
    N, H, d = 50, 2, 16
    L, q, k, v = _rand_case(N, 64, [4], H, d, seed=2)
    T = L["T"]
    heads = np.repeat(np.arange(H), T)
    rows = np.tile(np.arange(T), H)
    o, _ = fo.attn_rows(q, k, v, L["keep"], L["win"], 0.3, heads, rows)
    ref = torch.nn.functional.scaled_dot_product_attention(
        *(x.to(torch.float64) for x in (q, k, v)), is_causal=True, scale=0.3)
    np.testing.assert_allclose(o.reshape(H, T, d), ref.numpy(), rtol=0, atol=1e-12)


def test_tail_covering_every_base_is_causal_over_augmented():
    """With a boundary tail at least as long as every window, every row is kept,
    so every row sees all earlier rows: causal attention over the augmented
    sequence (library SDPA, fp64)."""
    N, W, H, d = 70, 16, 2, 16
    L, q, k, v = _rand_case(N, W, [3], H, d, seed=9, tail=W)
    T = L["T"]
    assert L["R"] == T
    o, lse = fo.attn_rows(q, k, v, L["keep"], L["win"], 0.4, np.repeat(np.arange(H), T), np.tile(np.arange(T), H))
    ref = torch.nn.functional.scaled_dot_product_attention(
        *(x.to(torch.float64) for x in (q, k, v)), is_causal=True, scale=0.4)
    np.testing.assert_allclose(o.reshape(H, T, d), ref.numpy(), rtol=0, atol=1e-12)


def test_softmax_rows_sum_to_one():
    """V = 1 everywhere => every output is sum(p)/l = 1 (rows of P sum to 1)."""
    L, q, k, _ = _rand_case(300, 40, [7], 2, 16, seed=4, std=3.0)
    v = torch.ones_like(k)
    T = L["T"]
    heads = np.repeat(np.arange(2), T)
    rows = np.tile(np.arange(T), 2)
    o, _ = fo.attn_rows(q, k, v, L["keep"], L["win"], 1.0, heads, rows)
    assert np.abs(o - 1.0).max() <= 1e-12


def test_lse_of_zero_scores_counts_visible_keys():
    """q = 0 => all scores 0 => LSE_i = ln |visible(i)| = ln(R_w + a + 1), with R_w
    the summaries retained before window w and a the in-window offset of row i."""
    N, W, ks = 500, 60, [1, 7, 13, 60, 100]
    M = _ceil(N, W)
    kk = inputs.k_schedule(M, ks, seed=8)
    L = fo.layout(N, W, kk)
    T = L["T"]
    q = torch.zeros((1, T, 8), dtype=torch.bfloat16)
    _, k, v = inputs.qkv((1, T, 8), seed=9)
    o, lse = fo.attn_rows(q, k, v, L["keep"], L["win"], 1.0, np.zeros(T, np.int64), np.arange(T))
    w = L["win"]
    count = L["ring_off"][w] + (np.arange(T) - L["win_off"][w]) + 1
    np.testing.assert_allclose(lse, np.log(count), rtol=0, atol=1e-12)


def test_first_row_sees_only_itself():
    L, q, k, v = _rand_case(30, 10, [3], 1, 8, seed=6)
    o, lse = fo.attn_rows(q, k, v, L["keep"], L["win"], 0.5, [0], [0])
    assert np.array_equal(o[0], _f64(v)[0, 0])
    assert lse[0] == pytest.approx(0.5 * float(_f64(q)[0, 0] @ _f64(k)[0, 0]), abs=1e-14)


# ----------------------------------------------------------------------------- retention / sequential


@pytest.mark.parametrize("N,W,ks,tail", [(700, 100, [10], 0), (1024, 100, [7, 30, 100], 0), (333, 50, [1, 51], 0),
                                         (90, 200, [4], 0), (700, 100, [10], 3), (333, 50, [1, 51], 60)])
def test_sequential_equals_masked_parallel(N, W, ks, tail):
    """App. A.1: sequential windows with KV dropping == masked-parallel."""
    H, d = 2, 16
    L, q, k, v = _rand_case(N, W, ks, H, d, seed=N, tail=tail)
    T = L["T"]
    for h in range(H):
        o_s, lse_s, rk, rv = fo.prefill_sequential(q[h], k[h], v[h], L["win_off"], L["keep"], 0.25)
        o_p, lse_p = fo.attn_rows(q, k, v, L["keep"], L["win"], 0.25, np.full(T, h), np.arange(T))
        np.testing.assert_allclose(o_s, o_p, rtol=0, atol=1e-12)
        np.testing.assert_allclose(lse_s, lse_p, rtol=0, atol=1e-12)
        # retained KV == the FOCUS rows, bit for bit, count == sum_w B_w
        kb = k[h].view(torch.int16).numpy().view(np.uint16)
        vb = v[h].view(torch.int16).numpy().view(np.uint16)
        assert rk.shape[0] == L["R"]
        assert np.array_equal(rk, kb[L["sum_idx"]]) and np.array_equal(rv, vb[L["sum_idx"]])


def test_retained_count_after_n_windows():
    """After n full windows with k | W the ring holds n*W/k summaries per head."""
    W, k, H, d = 200, 20, 1, 8
    for n in (1, 2, 5):
        L, q, kk, v = _rand_case(n * W, W, [k], H, d, seed=n)
        _, _, rk, _ = fo.prefill_sequential(q[0], kk[0], v[0], L["win_off"], L["keep"], 1.0,
                                            want=np.zeros(L["M"]))
        assert rk.shape[0] == n * W // k


# ----------------------------------------------------------------------------- decode


def test_decode_equals_prefill_row():
    """A decode step with the ring = retained summaries of earlier windows and the
    window buffer = earlier rows of the current window reproduces prefill row t."""
    N, W, ks, H, d = 900, 100, [9], 2, 16
    L, q, k, v = _rand_case(N, W, ks, H, d, seed=12)
    rng = np.random.default_rng(0)
    ts = rng.integers(0, L["T"], size=24)
    for h in range(H):
        o_p, lse_p = fo.attn_rows(q, k, v, L["keep"], L["win"], 0.2, np.full(ts.size, h), ts)
        for r, t in enumerate(ts):
            w = L["win"][t]
            ring_rows = L["sum_idx"][: L["ring_off"][w]]
            a = L["win_off"][w]
            ring_k = k[h][ring_rows][None] if ring_rows.size else torch.zeros((1, 1, d), dtype=torch.bfloat16)
            ring_v = v[h][ring_rows][None] if ring_rows.size else torch.zeros((1, 1, d), dtype=torch.bfloat16)
            wk = k[h][a:t][None] if t > a else torch.zeros((1, 1, d), dtype=torch.bfloat16)
            wv = v[h][a:t][None] if t > a else torch.zeros((1, 1, d), dtype=torch.bfloat16)
            o_d, lse_d = fo.decode(q[h][t][None], k[h][t][None], v[h][t][None], ring_k, ring_v,
                                   [ring_rows.size], wk, wv, [t - a], 0.2)
            np.testing.assert_allclose(o_d[0], o_p[r], rtol=0, atol=1e-12)
            assert abs(lse_d[0] - lse_p[r]) <= 1e-12


def test_decode_ring_order_is_irrelevant():
    n, R, F, d = 3, 57, 11, 32
    g = torch.Generator().manual_seed(1)
    ring_k, ring_v = (torch.randn((n, R, d), generator=g).bfloat16() for _ in range(2))
    win_k, win_v = (torch.randn((n, F, d), generator=g).bfloat16() for _ in range(2))
    q, kn, vn = (torch.randn((n, d), generator=g).bfloat16() for _ in range(3))
    o1, l1 = fo.decode(q, kn, vn, ring_k, ring_v, [R] * n, win_k, win_v, [F] * n, 0.3)
    perm = torch.randperm(R, generator=g)
    o2, l2 = fo.decode(q, kn, vn, ring_k[:, perm], ring_v[:, perm], [R] * n, win_k, win_v, [F] * n, 0.3)
    np.testing.assert_allclose(o1, o2, rtol=0, atol=1e-12)
    np.testing.assert_allclose(l1, l2, rtol=0, atol=1e-12)


# ----------------------------------------------------------------------------- k-mer-local visibility (main text)

def _local_case(N, W, ks, H, d, seed, std=1.0):
    M = _ceil(N, W)
    k = inputs.k_schedule(M, ks, seed=seed)
    L = fo.layout(N, W, k)
    L["k"] = k
    L["kmer"] = fo.layout_kmer(N, W, k)
    q, kk, v = inputs.qkv((H, L["T"], d), std=std, seed=seed)
    return L, q, kk, v


def _local(q, k, v, L, scale, heads, rows):
    return fo.attn_rows_kmer_local(q, k, v, L["kind"], L["win"], L["kmer"], scale, heads, rows)


@pytest.mark.parametrize("N,W,ks", LAYOUT_CASES)
def test_kmer_ids_closed_form(N, W, ks):
    """A window's rows come in blocks of k + 1 (k bases, then their FOCUS token),
    the last block possibly shorter: row at in-window offset a belongs to k-mer
    floor(a / (k + 1)); a window without summaries is one block."""
    M = _ceil(N, W)
    k = inputs.k_schedule(M, ks, seed=5)
    L = fo.layout(N, W, k)
    km = fo.layout_kmer(N, W, k)
    w = L["win"]
    a = np.arange(L["T"]) - L["win_off"][w]
    kw = k[w].astype(np.int64)
    expect = np.where(kw > 0, a // np.maximum(kw + 1, 1), 0)
    assert np.array_equal(km, expect)


def test_kmer_local_lse_of_zero_scores_counts_visible_keys():
    """q = 0 => LSE_i = ln |visible(i)|. Under the main-text rule a row at offset
    a of k-mer c (= a // (k+1)) of window w sees the a - c(k+1) + 1 rows of its
    k-mer up to itself, the c FOCUS rows of the earlier k-mers of its window, and
    the carried boundary when window w-1 has a FOCUS row (k_{w-1} > 0)."""
    N, W, ks = 700, 60, [1, 7, 13, 0, 60, 100]
    M = _ceil(N, W)
    kk = inputs.k_schedule(M, ks, seed=8)
    L = fo.layout(N, W, kk)
    km = fo.layout_kmer(N, W, kk)
    T = L["T"]
    q = torch.zeros((1, T, 8), dtype=torch.bfloat16)
    _, k, v = inputs.qkv((1, T, 8), seed=9)
    _, lse = fo.attn_rows_kmer_local(q, k, v, L["kind"], L["win"], km, 1.0, np.zeros(T, np.int64), np.arange(T))
    w = L["win"]
    a = np.arange(T) - L["win_off"][w]
    kw = kk[w].astype(np.int64)
    c = np.where(kw > 0, a // np.maximum(kw + 1, 1), 0)
    in_kmer = a - c * (kw + 1) + 1
    boundary = (w >= 1) & (kk[np.maximum(w - 1, 0)] > 0)
    count = in_kmer + c + boundary
    np.testing.assert_allclose(lse, np.log(count), rtol=0, atol=1e-12)


@pytest.mark.parametrize("k", [0, 64, 1_000])
def test_kmer_local_single_kmer_window_is_causal(k):
    """One window whose only k-mer spans it (k = 0, or k >= N): every row sees
    every earlier row, i.e. causal attention over the augmented sequence
    (library SDPA, fp64)."""
    N, H, d = 57, 2, 16
    L, q, kk, v = _local_case(N, 64, [k], H, d, seed=21)
    T = L["T"]
    o, lse = _local(q, kk, v, L, 0.35, np.repeat(np.arange(H), T), np.tile(np.arange(T), H))
    ref = torch.nn.functional.scaled_dot_product_attention(
        *(x.to(torch.float64) for x in (q, kk, v)), is_causal=True, scale=0.35)
    np.testing.assert_allclose(o.reshape(H, T, d), ref.numpy(), rtol=0, atol=1e-12)


def test_kmer_local_equals_appendix_mask_for_two_single_kmer_windows():
    """With k >= W every window is one k-mer closed by one FOCUS row; with two
    windows the only retained row before window 1 is window 0's FOCUS row, which
    is also the carried boundary, so both visibility rules give the same sets
    (the appendix form is pinned independently above)."""
    N, W, H, d = 90, 50, 2, 16
    L, q, kk, v = _local_case(N, W, [50], H, d, seed=22)
    assert L["M"] == 2 and L["R"] == 2
    T = L["T"]
    heads, rows = np.repeat(np.arange(H), T), np.tile(np.arange(T), H)
    o1, l1 = _local(q, kk, v, L, 0.25, heads, rows)
    o2, l2 = fo.attn_rows(q, kk, v, L["keep"], L["win"], 0.25, heads, rows)
    np.testing.assert_allclose(o1, o2, rtol=0, atol=1e-13)
    np.testing.assert_allclose(l1, l2, rtol=0, atol=1e-13)


def _perturb_rows(x, rows, seed):
    y = x.clone()
    g = torch.Generator().manual_seed(seed)
    y[:, rows] = torch.randn(y[:, rows].shape, generator=g).to(y.dtype) * 3
    return y


def test_kmer_local_invisible_rows_do_not_matter_and_visible_ones_do():
    """Main text: earlier windows' rows are reachable only through the carried
    boundary, and a row does not see the bases of other k-mers. Rewriting the
    K/V of every other earlier row leaves window w's outputs bit-identical;
    rewriting the boundary, or an earlier in-window FOCUS row, changes them."""
    N, W, H, d = 300, 60, 1, 16
    L, q, kk, v = _local_case(N, W, [10], H, d, seed=23)
    w = 3
    a, e = int(L["win_off"][w]), int(L["win_off"][w + 1])
    rows = np.arange(a, e)
    heads = np.zeros(rows.size, np.int64)
    o0, l0 = _local(q, kk, v, L, 0.25, heads, rows)
    prev = np.arange(int(L["win_off"][w - 1]), a)
    boundary = int(prev[L["kind"][prev] == 1][-1])
    assert boundary == a - 1
    hidden = [j for j in range(a) if j != boundary]
    # bases of the window's first k-mer are hidden from the rows of its later k-mers
    later = rows[L["kmer"][rows] >= 1]
    first_bases = [j for j in range(a, e) if L["kmer"][j] == 0 and L["kind"][j] == 0]
    o1, l1 = _local(_perturb_rows(q, [], 1), _perturb_rows(kk, hidden, 2), _perturb_rows(v, hidden, 3), L, 0.25,
                    heads, rows)
    assert np.array_equal(o0, o1) and np.array_equal(l0, l1)
    ol0, _ = _local(q, kk, v, L, 0.25, np.zeros(later.size, np.int64), later)
    ol1, _ = _local(q, _perturb_rows(kk, first_bases, 4), _perturb_rows(v, first_bases, 5), L, 0.25,
                    np.zeros(later.size, np.int64), later)
    assert np.array_equal(ol0, ol1)
    ob, _ = _local(q, _perturb_rows(kk, [boundary], 6), _perturb_rows(v, [boundary], 7), L, 0.25, heads, rows)
    assert np.abs(ob - o0).max(axis=1).min() > 0          # every row of window w sees the boundary
    first_focus = [j for j in range(a, e) if L["kmer"][j] == 0 and L["kind"][j] == 1]
    of, _ = _local(q, _perturb_rows(kk, first_focus, 8), _perturb_rows(v, first_focus, 9), L, 0.25,
                   np.zeros(later.size, np.int64), later)
    assert np.abs(of - ol0).max(axis=1).min() > 0         # every later k-mer sees the first FOCUS row


# ----------------------------------------------------------------------------- rotary position embedding

def _one_hot_bf16(d, idx):
    x = torch.zeros(d, dtype=torch.bfloat16)
    x[idx] = 1.0
    return x


@pytest.mark.parametrize("d", [8, 64, 128])
def test_rope_one_hot_closed_form(d):
    """RoFormer rotation, rotate-half pairing: e_i at position p goes to
    cos(p t_i) e_i + sin(p t_i) e_{i+d/2} and e_{i+d/2} to
    -sin(p t_i) e_i + cos(p t_i) e_{i+d/2}, t_i = base^(-2i/d): t_0 = 1 and
    t_{d/4} = base^(-1/2)."""
    base, h = 10_000.0, d // 2
    for i, theta in ((0, 1.0), (d // 4, base ** -0.5), (h - 1, base ** (-2.0 * (h - 1) / d))):
        for p in (0, 1, 7, 123_457, 1_010_000):
            y = fo.rope(_one_hot_bf16(d, i), p, base)
            e = np.zeros(d)
            e[i], e[i + h] = math.cos(p * theta), math.sin(p * theta)
            np.testing.assert_allclose(y, e, rtol=0, atol=1e-12)
            y = fo.rope(_one_hot_bf16(d, i + h), p, base)
            e = np.zeros(d)
            e[i], e[i + h] = -math.sin(p * theta), math.cos(p * theta)
            np.testing.assert_allclose(y, e, rtol=0, atol=1e-12)


def test_rope_position_zero_is_identity_and_pairs_keep_their_norm():
    x = inputs.normal_bf16((50, 64), 1.0, seed=3)
    pos = np.arange(50) * 20_011
    np.testing.assert_array_equal(fo.rope(x, 0, 500_000.0), _f64(x))
    y = fo.rope(x, pos, 500_000.0)
    xf = _f64(x)
    np.testing.assert_allclose(y[:, :32] ** 2 + y[:, 32:] ** 2, xf[:, :32] ** 2 + xf[:, 32:] ** 2, rtol=1e-13, atol=0)


def test_rope_attention_depends_only_on_relative_positions():
    """<R(p) q, R(p') k> depends on p - p' only, so adding one offset to every
    position leaves the attention outputs unchanged."""
    L, q, k, v = _rand_case(300, 60, [7], 2, 32, seed=12)
    T = L["T"]
    heads, rows = np.repeat(np.arange(2), T), np.tile(np.arange(T), 2)
    outs = []
    for shift in (0, 987_654):
        pos = np.arange(T) + shift
        qf = fo.rope(q, pos, 10_000.0)
        kf = fo.rope(k, pos, 10_000.0)
        outs.append(fo.attn_rows_f64(qf, kf, v, L["keep"], L["win"], 0.2, heads, rows))
    np.testing.assert_allclose(outs[0][0], outs[1][0], rtol=0, atol=1e-9)
    np.testing.assert_allclose(outs[0][1], outs[1][1], rtol=0, atol=1e-9)


def test_fp64_attention_variants_equal_the_pinned_bf16_ones():
    """attn_rows_f64 / decode_f64 on the exactly widened bf16 inputs equal
    attn_rows / decode (pinned above) to the last bit of fp64 arithmetic."""
    L, q, k, v = _rand_case(400, 50, [1, 10, 60], 2, 16, seed=13)
    T = L["T"]
    heads, rows = np.repeat(np.arange(2), T), np.tile(np.arange(T), 2)
    o1, l1 = fo.attn_rows(q, k, v, L["keep"], L["win"], 0.3, heads, rows)
    o2, l2 = fo.attn_rows_f64(_f64(q), _f64(k), v, L["keep"], L["win"], 0.3, heads, rows)
    np.testing.assert_allclose(o1, o2, rtol=0, atol=1e-15)
    np.testing.assert_allclose(l1, l2, rtol=0, atol=1e-14)
    n, d, C = 3, 16, 20
    qn, kn, vn = inputs.qkv((n, d), seed=14)
    rk, rv, wk = inputs.qkv((n, C, d), seed=15)
    wv = inputs.normal_bf16((n, C, d), 1.0, seed=16)
    R, fill = np.array([0, 5, 20]), np.array([3, 0, 19])
    a = fo.decode(qn, kn, vn, rk, rv, R, wk, wv, fill, 0.25)
    b = fo.decode_f64(_f64(qn), _f64(kn), vn, _f64(rk), rv, R, _f64(wk), wv, fill, 0.25)
    np.testing.assert_allclose(a[0], b[0], rtol=0, atol=1e-15)
    np.testing.assert_allclose(a[1], b[1], rtol=0, atol=1e-14)


def test_round_bf16_is_nearest_even_and_matches_torch():
    """Ties go to the even significand (1 + 2^-8 lies halfway between 1 and
    1 + 2^-7); otherwise the nearest bf16 value, as torch's fp32 -> bf16
    conversion gives for values that fp32 holds exactly."""
    assert fo.round_bf16(1.0 + 2.0 ** -8) == 1.0
    assert fo.round_bf16(1.0 + 3 * 2.0 ** -8) == 1.0 + 2.0 ** -6
    assert fo.round_bf16(-(1.0 + 3 * 2.0 ** -8)) == -(1.0 + 2.0 ** -6)
    assert fo.round_bf16(1.0 + 2.0 ** -8 + 2.0 ** -30) == 1.0 + 2.0 ** -7
    x = inputs.normal_bf16((2000,), 3.0, seed=9).float() * (1 + 1e-3)
    ref = x.to(torch.bfloat16).double().numpy()
    got = np.array([fo.round_bf16(float(v)) for v in x.double().numpy()])
    np.testing.assert_array_equal(got, ref)


def test_rope_rounded_is_the_rounded_exact_rotation():
    x = inputs.normal_bf16((40, 64), 1.0, seed=10)
    pos = np.arange(40) * 9_973
    y = fo.rope(x, pos, 10_000.0)
    yr = fo.rope(x, pos, 10_000.0, round_bf16=True)
    np.testing.assert_array_equal(yr, np.vectorize(fo.round_bf16)(y))
    assert (np.abs(yr - y) <= 2.0 ** -8 * np.abs(y)).all()     # half a step of 8 significant bits


# ----------------------------------------------------------------------------- adaptive windows (W per window)

SCHED_CASES = [
    (2_500, [400, 1_000, 100, 1_000], [10, 25, 7, 200]),
    (1_037, [64, 1_000, 1_000], [8, 100, 3]),          # the last window is partial; the third is never reached
    (37, [1, 2, 3, 50], [1, 1, 2, 9]),
    (300, [128, 64, 32, 16, 8, 52], [0, 5, 32, 1, 9, 13]),
]


@pytest.mark.parametrize("N,Ws,ks", SCHED_CASES)
def test_adaptive_windows_sizes_and_offsets_closed_form(N, Ws, ks):
    """Adaptive windowing (Sec. 5: W and k chosen per region): window w holds
    the next W_w bases (the last one what is left); T = N + sum ceil(n_w/k_w),
    R = sum B_w, and base_off is the running sum of the window lengths."""
    cuts = _cuts(N, Ws)
    M = len(cuts) - 1
    k = np.asarray(ks[:M], np.int32)
    T, R, M2 = fo.layout_size(N, Ws, k)
    assert M2 == M
    n_w = np.diff(cuts)
    B_w = [(_ceil(int(n), int(kk)) if kk > 0 else 0) for n, kk in zip(n_w, k)]
    assert (R, T) == (sum(B_w), N + sum(B_w))
    L = fo.layout(N, Ws, k)
    assert np.array_equal(L["base_off"], cuts)
    assert np.array_equal(np.diff(L["win_off"]), n_w + np.array(B_w))


@pytest.mark.parametrize("N,Ws,ks", SCHED_CASES)
@pytest.mark.parametrize("close_tail", [True, False])
def test_adaptive_windows_match_string_construction(N, Ws, ks, close_tail):
    M = len(_cuts(N, Ws)) - 1
    k = np.asarray(ks[:M], np.int32)
    nt = inputs.nucleotides(1, N, seed=12).numpy()
    L = fo.layout(N, Ws, k, nt=nt, close_tail=close_tail)
    seq = "".join("ACGT"[x] for x in nt[0])
    assert "".join("ACGTS"[x] for x in L["tok"][0]) == _string_layout(seq, Ws, k, close_tail)
    km = fo.layout_kmer(N, Ws, k, close_tail=close_tail)
    w = L["win"]
    a = np.arange(L["T"]) - L["win_off"][w]
    kw = k[w].astype(np.int64)
    assert np.array_equal(km, np.where(kw > 0, a // np.maximum(kw + 1, 1), 0))


@pytest.mark.parametrize("tail", [0, 3])
def test_adaptive_windows_attention_matches_streaming_simulation(tail):
    N, Ws, ks, H, d = 300, [128, 64, 32, 16, 8, 52], [0, 5, 32, 1, 9, 13], 2, 16
    L = fo.layout(N, Ws, ks, tail=tail)
    q, k, v = inputs.qkv((H, L["T"], d), seed=77)
    T = L["T"]
    heads, rows = np.repeat(np.arange(H), T), np.tile(np.arange(T), H)
    o, lse = fo.attn_rows(q, k, v, L["keep"], L["win"], 0.25, heads, rows)
    vis = _visible_sets_by_streaming(L, tail)
    qd, kd, vd = _f64(q), _f64(k), _f64(v)
    for r, (h, i) in enumerate(zip(heads, rows)):
        j = np.array(vis[i])
        sc = 0.25 * (kd[h, j] @ qd[h, i])
        np.testing.assert_allclose(o[r], scipy.special.softmax(sc) @ vd[h, j], rtol=0, atol=1e-12)
        assert abs(lse[r] - scipy.special.logsumexp(sc)) <= 1e-12 * max(1.0, abs(lse[r]))


def test_window_schedule_must_cover_the_sequence():
    with pytest.raises(ValueError):
        fo.layout_size(100, [30, 30], [5])


# ----------------------------------------------------------------------------- token embedding (Sec. 3.2)

def test_embed_tokens_one_hot_table_spells_the_string_layout():
    """With a table whose row j is the one-hot vector of j (bf16 1.0 = 0x3F80),
    each output row names its token, so the rows spell the independent string
    construction of the layout (a summary 'S' after every k bases)."""
    N, W, ks = 777, 100, [7, 30, 100]
    M = _ceil(N, W)
    k = inputs.k_schedule(M, ks, seed=5)
    nt = inputs.nucleotides(2, N, seed=13).numpy()
    L = fo.layout(N, W, k, nt=nt)
    n_tok, D = 5, 8
    table = np.zeros((n_tok, D), np.uint16)
    table[np.arange(n_tok), np.arange(n_tok)] = 0x3F80
    out = fo.embed_tokens(L["tok"], table)
    assert out.shape == (2, L["T"], D)
    for b in range(2):
        got = "".join("ACGTS"[int(np.argmax(r))] for r in out[b])
        assert got == _string_layout("".join("ACGT"[x] for x in nt[b]), W, k, True)
        assert (out[b][:, n_tok:] == 0).all() and (out[b] != 0).sum() == L["T"]


def test_embed_tokens_summary_rows_sit_at_summary_positions():
    """The summary token's vector appears exactly on the layout's summary rows,
    T - N of them (T = N + sum_w ceil(n_w / k_w), App. A), and nucleotide rows
    carry their base's vector."""
    N, W, ks = 4_000, 1_000, [100]
    M = _ceil(N, W)
    k = inputs.k_schedule(M, ks, seed=1)
    nt = inputs.nucleotides(1, N, seed=3).numpy()
    L = fo.layout(N, W, k, nt=nt)
    rng = np.random.default_rng(0)
    table = rng.integers(0, 1 << 16, size=(5, 64), dtype=np.uint16)
    out = fo.embed_tokens(L["tok"], table)[0]
    is_summary = (out == table[fo.SUMMARY_TOKEN]).all(axis=1)
    assert is_summary.sum() == L["T"] - N == M * _ceil(W, 100)
    assert np.array_equal(is_summary, L["kind"] == 1)
    base_rows = np.flatnonzero(L["kind"] == 0)
    assert np.array_equal(out[base_rows], table[nt[0][L["src"][base_rows]]])


def test_embed_tokens_out_of_table_token_is_a_zero_row():
    table = np.full((5, 8), 0x3F80, np.uint16)
    out = fo.embed_tokens(np.array([0, 9, 4], np.uint8), table)
    assert (out[1] == 0).all() and (out[0] == 0x3F80).all() and (out[2] == 0x3F80).all()
