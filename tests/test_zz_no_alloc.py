"""focus_attn_decode_noalloc: the decode entry point for callers that cannot
give the library device scratch (a plugin inside a runtime that owns all
device memory, a serving loop that must not call cudaMalloc/cudaFree between
steps). It must give the same results as focus_attn_decode with a caller
workspace, on consecutive calls, and refuse caches that need more scratch than
its fixed array holds.

The file name sorts last so that a run stopping at the first failure has run
every other test first.
"""
import ctypes
import math

import numpy as np
import pytest
import torch

from paper_2511_14694_gb300 import focus, inputs

pytestmark = pytest.mark.gpu


def _cache_pair(B, H, d, R, fill, C_ring, C_win, W, k, g, rope):
    caches = []
    for _ in range(2):
        c = focus.Cache(B, H, d, C_ring=C_ring, C_win=C_win, W=W, k_sched=[k] * 64, q_per_kv=g, rope_theta=rope)
        for i, t in enumerate((c.ring_k, c.ring_v, c.win_k, c.win_v)):
            t.copy_(inputs.normal_bf16(t.shape, 1.0, seed=70 + i, device="cuda"))
        c.ring_len.fill_(R)
        c.win_idx.fill_(3)
        c.win_fill.copy_(torch.from_numpy(np.asarray(fill, np.int32)))
        c.pos_base.fill_(3 * (W + -(-W // k)))
        caches.append(c)
    return caches


# (query heads per K/V head, rotary base): the CUDA-core split kernel without
# rotation, and the grouped-query tensor-core kernel with the rotated q/k rows
# that the library also keeps in its fixed array
@pytest.mark.parametrize("g,rope", [(1, 0.0), (4, 1e4)])
def test_noalloc_decode_matches_workspace_decode_on_consecutive_calls(g, rope):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    focus.device_status(clear=True)
    B, H, d, W, k = 8, 4, 128, 1_000, 100
    fill = [0, 5, 1_008, 1_009, 300, 999, 17, 640]        # two sequences finish their window
    ref, noalloc = _cache_pair(B, H, d, 2_000, fill, C_ring=2_100, C_win=1_024, W=W, k=k, g=g, rope=rope)
    assert ref.workspace_bytes() <= (16 << 20)
    ws = ref.new_workspace()
    for step in range(2):
        q = inputs.normal_bf16((B, H * g, d), 1.0, seed=500 + step, device="cuda")
        kn = inputs.normal_bf16((B, H, d), 1.0, seed=600 + step, device="cuda")
        vn = inputs.normal_bf16((B, H, d), 1.0, seed=700 + step, device="cuda")
        o_ref, lse_ref = focus.attn_decode(ref, q, kn, vn, workspace=ws)
        focus.kv_compact_window(ref)
        o_na, lse_na = focus.attn_decode_noalloc(noalloc, q, kn, vn)
        focus.kv_compact_window(noalloc)
        torch.cuda.synchronize()
        err = (o_na.float() - o_ref.float()).abs().max().item()
        lerr = ((lse_na - lse_ref).abs() / lse_ref.abs().clamp(min=1.0)).max().item()
        assert err <= 2e-2 and lerr <= 1e-3, (step, err, lerr)
        for a, b in ((ref.ring_len, noalloc.ring_len), (ref.win_fill, noalloc.win_fill),
                     (ref.win_idx, noalloc.win_idx), (ref.pos_base, noalloc.pos_base)):
            assert torch.equal(a, b)
    assert torch.equal(ref.ring_k, noalloc.ring_k) and torch.equal(ref.win_k, noalloc.win_k)
    assert torch.equal(ref.win_v, noalloc.win_v)
    assert focus.device_status(clear=True) == 0


def test_noalloc_decode_refuses_caches_beyond_its_scratch():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    # 64 x 32 heads x d=128 with 40k ring rows needs ~42 MB of partials > 16 MiB
    c = focus.CacheDesc()
    c.B, c.H, c.d, c.C_ring, c.C_win, c.W, c.n_windows = 64, 32, 128, 40_000, 1_024, 1_000, 1
    dummy = torch.zeros(16, dtype=torch.int32, device="cuda")
    for f in ("ring_k", "ring_v", "win_k", "win_v", "ring_len", "win_fill", "win_idx", "k_per_window"):
        setattr(c, f, dummy.data_ptr())
    lib = focus.load()
    assert lib.focus_decode_workspace_size(ctypes.byref(c)) > (16 << 20)
    p = dummy.data_ptr()
    rc = lib.focus_attn_decode_noalloc(ctypes.byref(c), p, p, p, 1.0 / math.sqrt(128), p, None, None)
    assert rc == 3   # FOCUS_ERR_CAPACITY, nothing launched
