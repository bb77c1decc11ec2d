"""The masked-parallel prefill from pinned host memory (focus_prefill_host,
through pipeline.prefill_masked_parallel_host) runs the same kernels per group of heads or
sequences, with the copies on side streams: its outputs must equal, bit for bit,
those of the all-at-once device path on the same inputs, and the ring must hold
the same rows."""
from __future__ import annotations

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


@pytest.mark.parametrize("B,H,d,g,groups,rope,local", [(1, 4, 64, 1, 3, 0.0, False), (3, 2, 128, 1, 2, 0.0, False),
                                                       (1, 2, 128, 2, 2, 0.0, False), (2, 2, 64, 1, 8, 0.0, False),
                                                       (1, 4, 128, 1, 2, 10_000.0, False),
                                                       (1, 4, 128, 2, 2, 10_000.0, False),
                                                       (2, 2, 64, 1, 2, 0.0, True), (1, 4, 128, 1, 4, 10_000.0, True)])
def test_host_pipeline_matches_device_path(B, H, d, g, groups, rope, local):
    """The host-buffer entry point gives the device path's outputs and ring bit for
    bit, with grouped heads, the rotary embedding (a pass per part, or the
    persistent kernel rotating in place for grouped heads) and the k-mer-local
    mask; the workspace sized for the whole cache serves every part in turn."""
    N, W = 5_000, 1_000
    k = inputs.k_schedule(-(-N // W), [100, 10, 50], seed=3)
    L_dev = focus.layout_alloc(N, W, k, B=B)
    L_host = focus.layout_alloc(N, W, k, B=B)
    nt = inputs.nucleotides(B, N, seed=5, device="cuda")
    T = L_dev["T"]
    q, kk, v = inputs.qkv((B, H * g, T, d), std=1.0, seed=7, device="cuda", q_per_kv=g)
    # the device path
    focus.layout_run(L_dev, nt)
    c_dev = focus.Cache(B, H, d, C_ring=L_dev["R"], k_sched=k, q_per_kv=g, rope_theta=rope)
    fl = focus.PREFILL_KMER_LOCAL if local else 0
    o_dev, lse_dev = pipeline.prefill_masked_parallel(c_dev, q, kk, v, L_dev, flags=fl)
    # the host path
    pin = lambda t: t.cpu().pin_memory()                                  # noqa: E731
    host = dict(nt=pin(nt), q=pin(q), k=pin(kk), v=pin(v), o=torch.empty(q.shape, dtype=torch.bfloat16).pin_memory(),
                lse=torch.empty((B, H * g, T), dtype=torch.float32).pin_memory())
    dev = dict(nt=torch.empty_like(nt), q=torch.empty_like(q), k=torch.empty_like(kk), v=torch.empty_like(v),
               o=torch.empty_like(q), lse=torch.empty((B, H * g, T), dtype=torch.float32, device="cuda"))
    c_host = focus.Cache(B, H, d, C_ring=L_host["R"], k_sched=k, q_per_kv=g, rope_theta=rope)
    pipeline.prefill_masked_parallel_host(c_host, L_host, host, dev, groups=groups, flags=fl)
    torch.cuda.synchronize()
    assert np.array_equal(bits(host["o"]), bits(o_dev))
    assert np.array_equal(host["lse"].numpy(), lse_dev.cpu().numpy())
    assert np.array_equal(L_host["win_off"].cpu().numpy(), L_dev["win_off"].cpu().numpy())
    assert np.array_equal(bits(c_host.ring_k), bits(c_dev.ring_k))
    assert np.array_equal(bits(c_host.ring_v), bits(c_dev.ring_v))
    assert np.array_equal(c_host.ring_len.cpu().numpy(), c_dev.ring_len.cpu().numpy())
