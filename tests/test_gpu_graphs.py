"""CUDA-graph capture of the library's entry points: the layout, the
masked-parallel prefill (bulk compaction + attention), decode steps with window
roll-overs, the allocation-free decode and the token-embedding gather, captured
once and replayed, give the eager calls' results bit for bit (the entry points
enqueue work on the given stream only, allocate nothing and never synchronize).
The streaming prefill's graph is covered in test_gpu_parity.py."""
import numpy as np
import pytest
import torch

from paper_2511_14694_gb300 import focus, inputs, pipeline
from test_gpu_parity import bits

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _clean_status():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    focus.device_status(clear=True)
    yield
    assert focus.device_status(clear=True) == 0, "a kernel reported an error"


def _capture(fn):
    """fn() once eagerly (the library's one-time set-up), then captured."""
    fn()
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        fn()
    torch.cuda.synchronize()
    return g


def test_layout_graph_replay():
    N, W = 7_777, 1_000
    k_s = inputs.k_schedule(-(-N // W), [10, 100, 7], seed=3)
    nt = inputs.nucleotides(2, N, seed=4, device="cuda")
    ref = focus.layout(N, W, k_s, nt=nt)
    L = focus.layout_alloc(N, W, k_s, 2, True, "cuda", 0)
    g = _capture(lambda: focus.layout_run(L, nt))
    names = ("kind", "src", "pos", "win", "keep", "win_off", "ring_off", "base_off", "tok", "sum_idx")
    for name in names:
        L[name].zero_()
    g.replay()
    torch.cuda.synchronize()
    for name in names:
        assert torch.equal(L[name], ref[name]), name


def test_masked_parallel_prefill_graph_replay():
    N, W, B, H, d = 20_000, 1_000, 2, 4, 128
    k_s = inputs.k_schedule(-(-N // W), [100, 50], seed=6)
    L = focus.layout(N, W, k_s)
    q, k, v = inputs.qkv((B, H, L["T"], d), seed=7, device="cuda")
    c_e = focus.Cache(B, H, d, C_ring=L["R"])
    o_e, l_e = pipeline.prefill_masked_parallel(c_e, q, k, v, L)
    c_g = focus.Cache(B, H, d, C_ring=L["R"])
    o_g, l_g = torch.empty_like(q), torch.empty_like(l_e)
    g = _capture(lambda: pipeline.prefill_masked_parallel(c_g, q, k, v, L, o=o_g, lse=l_g))
    for t in (o_g, l_g, c_g.ring_k, c_g.ring_v):
        t.zero_()
    g.replay()
    torch.cuda.synchronize()
    assert np.array_equal(bits(o_g), bits(o_e))
    assert torch.equal(l_g, l_e)
    assert np.array_equal(bits(c_g.ring_k), bits(c_e.ring_k))


@pytest.mark.parametrize("g_heads,rope", [(1, 0.0), (4, 0.0), (1, 10_000.0)])
def test_decode_step_graph_replay(g_heads, rope):
    """One decode step (attention + window roll-over) captured with static
    q/k_new/v_new buffers; each step copies its token into them and replays. The
    cache's lengths live in device memory, so every replay advances them; 60
    steps with windows of 50 rows cross roll-overs."""
    B, H, d, W, steps = 3, 2, 64, 50, 60
    k_sched = np.array([10, 7, 25, 50, 3, 10, 10, 10], np.int32)
    caches = [focus.Cache(B, H, d, C_ring=512, C_win=72, W=W, k_sched=k_sched, q_per_kv=g_heads, rope_theta=rope)
              for _ in range(2)]
    gen = torch.Generator(device="cuda").manual_seed(13)
    for t in (caches[0].ring_k, caches[0].ring_v, caches[0].win_k, caches[0].win_v):
        t.copy_(torch.randn(t.shape, generator=gen, device="cuda").bfloat16())
    for a, b in zip((caches[0].ring_k, caches[0].ring_v, caches[0].win_k, caches[0].win_v),
                    (caches[1].ring_k, caches[1].ring_v, caches[1].win_k, caches[1].win_v)):
        b.copy_(a)
    for c in caches:
        c.ring_len.copy_(torch.tensor([0, 37, 300], dtype=torch.int32))
        c.win_idx.copy_(torch.tensor([0, 1, 2], dtype=torch.int32))
        c.win_fill.copy_(torch.tensor([0, 49, 20], dtype=torch.int32))
    qs = inputs.normal_bf16((steps, B, H * g_heads, d), 1.0, seed=21, device="cuda")
    ks = inputs.normal_bf16((steps, B, H, d), 1.0, seed=22, device="cuda")
    vs = inputs.normal_bf16((steps, B, H, d), 1.0, seed=23, device="cuda")
    # eager
    ce = caches[0]
    ws_e = ce.new_workspace()
    eager = []
    for s in range(steps):
        o, lse = focus.attn_decode(ce, qs[s], ks[s], vs[s], workspace=ws_e)
        focus.kv_compact_window(ce)
        eager.append((o.clone(), lse.clone()))
    # graph: static buffers, one step captured after a throw-away cache's eager call
    cg = caches[1]
    q_b, k_b, v_b = torch.empty_like(qs[0]), torch.empty_like(ks[0]), torch.empty_like(vs[0])
    o_b = torch.empty_like(q_b)
    l_b = torch.empty((B, H * g_heads), dtype=torch.float32, device="cuda")
    ws_g = cg.new_workspace()
    warm = focus.Cache(B, H, d, C_ring=512, C_win=72, W=W, k_sched=k_sched, q_per_kv=g_heads, rope_theta=rope)
    focus.attn_decode(warm, q_b.zero_(), k_b.zero_(), v_b.zero_(), o=o_b, lse=l_b, workspace=warm.new_workspace())
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        focus.attn_decode(cg, q_b, k_b, v_b, o=o_b, lse=l_b, workspace=ws_g)
        focus.kv_compact_window(cg)
    for s in range(steps):
        q_b.copy_(qs[s])
        k_b.copy_(ks[s])
        v_b.copy_(vs[s])
        graph.replay()
        torch.cuda.synchronize()
        assert np.array_equal(bits(o_b), bits(eager[s][0])), f"step {s}"
        assert torch.equal(l_b, eager[s][1]), f"step {s}"
    for a, b in ((ce.ring_len, cg.ring_len), (ce.win_fill, cg.win_fill), (ce.win_idx, cg.win_idx)):
        assert torch.equal(a, b)
    assert np.array_equal(bits(ce.ring_k), bits(cg.ring_k))
    assert np.array_equal(bits(ce.win_k), bits(cg.win_k))


def test_embed_tokens_graph_replay():
    N, W = 5_000, 1_000
    nt = inputs.nucleotides(1, N, seed=8, device="cuda")
    L = focus.layout(N, W, [100], nt=nt)
    table = inputs.normal_bf16((5, 512), 1.0, seed=9, device="cuda")
    ref = focus.embed_tokens(L["tok"], table)
    out = torch.empty_like(ref)
    g = _capture(lambda: focus.embed_tokens(L["tok"], table, out=out))
    out.zero_()
    g.replay()
    torch.cuda.synchronize()
    assert np.array_equal(bits(out), bits(ref))


def test_decode_noalloc_graph_replay():
    """The allocation-free decode (library-owned scratch) captured and replayed
    equals focus_attn_decode with a caller workspace."""
    B, H, d, W = 2, 4, 128, 50
    k_sched = np.full(64, 10, np.int32)
    caches = [focus.Cache(B, H, d, C_ring=256, C_win=64, W=W, k_sched=k_sched) for _ in range(2)]
    gen = torch.Generator(device="cuda").manual_seed(17)
    for t in (caches[0].ring_k, caches[0].ring_v, caches[0].win_k, caches[0].win_v):
        t.copy_(torch.randn(t.shape, generator=gen, device="cuda").bfloat16())
    for a, b in zip((caches[0].ring_k, caches[0].ring_v, caches[0].win_k, caches[0].win_v),
                    (caches[1].ring_k, caches[1].ring_v, caches[1].win_k, caches[1].win_v)):
        b.copy_(a)
    for c in caches:
        c.ring_len.fill_(100)
        c.win_idx.fill_(10)
        c.win_fill.fill_(7)
    q, kn, vn = (inputs.normal_bf16((B, H, d), 1.0, seed=30 + i, device="cuda") for i in range(3))
    o_e, l_e = focus.attn_decode(caches[0], q, kn, vn, workspace=caches[0].new_workspace())
    o_g = torch.empty_like(q)
    l_g = torch.empty((B, H), dtype=torch.float32, device="cuda")
    warm = focus.Cache(B, H, d, C_ring=256, C_win=64, W=W, k_sched=k_sched)
    focus.attn_decode_noalloc(warm, q, kn, vn, o=o_g, lse=l_g)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        focus.attn_decode_noalloc(caches[1], q, kn, vn, o=o_g, lse=l_g)
    o_g.zero_()
    g.replay()
    torch.cuda.synchronize()
    assert np.array_equal(bits(o_g), bits(o_e))
    assert torch.equal(l_g, l_e)
    assert torch.equal(caches[0].win_fill, caches[1].win_fill)
