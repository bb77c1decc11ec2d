"""Failure detection and checkpoint/resume on the GPU, without a fault:

- a bounded device wait that nothing completes gives up and reports
  FOCUS_ERR_TIMEOUT in the status word (focus_selftest_timeout, the same wait
  every kernel uses); while the word holds it, prefill kernels skip their work;
  once cleared, the context computes the right rows again;
- the decode cache is caller-owned state: a snapshot restored into the cache
  resumes decoding bit for bit."""
from __future__ import annotations

import math

import numpy as np
import pytest
import torch

from oracle import focus_oracle as fo
from paper_2511_14694_gb300 import focus, inputs, pipeline
from test_gpu_parity import assert_attn_close, bits

pytestmark = pytest.mark.gpu
FOCUS_ERR_TIMEOUT = 5


@pytest.fixture(autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    focus.device_status(clear=True)
    yield
    focus.device_status(clear=True)


def test_bounded_wait_times_out_and_the_context_stays_usable():
    N, W, B, H, d = 3_000, 1_000, 1, 2, 64
    L = focus.layout(N, W, [100])
    q, k, v = inputs.qkv((B, H, L["T"], d), seed=3, device="cuda")
    cache = focus.Cache(B, H, d, C_ring=L["R"])
    focus.kv_compact_bulk(cache, k, v, L)
    torch.cuda.synchronize()
    # the wait gives up after 20 ms and reports; nothing faults, nothing hangs
    focus.selftest_timeout(20_000_000)
    assert focus.device_status(clear=False) == FOCUS_ERR_TIMEOUT
    # while the word holds the timeout, a prefill launch skips its work
    o = torch.full_like(q, 7.0)
    lse = torch.full((B, H, L["T"]), 7.0, dtype=torch.float32, device="cuda")
    focus.attn_prefill(cache, q, k, v, L, o=o, lse=lse)
    torch.cuda.synchronize()
    assert bool((o == 7.0).all()) and bool((lse == 7.0).all())
    assert focus.device_status(clear=True) == FOCUS_ERR_TIMEOUT
    # cleared: the same call computes the right rows
    focus.attn_prefill(cache, q, k, v, L, o=o, lse=lse)
    torch.cuda.synchronize()
    assert focus.device_status(clear=True) == 0
    ref = fo.layout(N, W, [100])
    T = L["T"]
    heads, rows = np.repeat(np.arange(B * H), T), np.tile(np.arange(T), B * H)
    o_ref, lse_ref = fo.attn_rows(q.reshape(B * H, T, d).cpu(), k.reshape(B * H, T, d).cpu(),
                                  v.reshape(B * H, T, d).cpu(), ref["keep"], ref["win"], 1 / math.sqrt(d), heads, rows)
    assert_attn_close(o, lse, o_ref.reshape(B, H, T, d), lse_ref.reshape(B, H, T), "after the timeout")


@pytest.mark.parametrize("g,rope", [(1, 0.0), (4, 10_000.0)])
def test_decode_resumes_bit_identically_from_a_snapshot(g, rope):
    B, H, d, W = 3, 2, 128, 50
    k_sched = np.array([10, 25, 7, 50, 10, 10, 10, 10], np.int32)
    cache = focus.Cache(B, H, d, C_ring=256, C_win=64, W=W, k_sched=k_sched, q_per_kv=g, rope_theta=rope)
    gen = torch.Generator(device="cuda").manual_seed(9)
    for t in (cache.ring_k, cache.ring_v, cache.win_k, cache.win_v):
        t.copy_(torch.randn(t.shape, generator=gen, device="cuda").bfloat16())
    cache.ring_len.copy_(torch.tensor([0, 20, 130], dtype=torch.int32))
    cache.win_idx.copy_(torch.tensor([0, 1, 2], dtype=torch.int32))
    cache.win_fill.copy_(torch.tensor([0, 40, 3], dtype=torch.int32))
    steps = [(inputs.normal_bf16((B, H * g, d), 1.0, seed=100 + s, device="cuda"),
              inputs.normal_bf16((B, H, d), 1.0, seed=200 + s, device="cuda"),
              inputs.normal_bf16((B, H, d), 1.0, seed=300 + s, device="cuda")) for s in range(40)]

    def run(seq):
        outs = []
        for q, kn, vn in seq:
            o, lse = focus.attn_decode(cache, q, kn, vn)
            focus.kv_compact_window(cache)
            outs.append((o.clone(), lse.clone()))
        return outs

    run(steps[:15])                                   # into the stream, across window retirements
    snap = cache.snapshot()
    first = run(steps[15:])
    end_state = cache.snapshot()
    cache.restore(snap)                               # back to step 15
    second = run(steps[15:])
    torch.cuda.synchronize()
    assert focus.device_status(clear=True) == 0
    for (o1, l1), (o2, l2) in zip(first, second):
        assert np.array_equal(bits(o1), bits(o2)) and torch.equal(l1, l2)
    for n, t in cache.snapshot().items():
        assert torch.equal(t, end_state[n]), n
