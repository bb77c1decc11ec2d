"""GPU parity of focus_embed_tokens (the augmented sequence's input rows, Sec.
3.2 "Setup and tokens"): bit-exact against the oracle's table lookup on the
device layout's token stream, ragged widths, an out-of-table token, and sampled
rows of the 128 kb layout at an Evo-2-7B-like width of 4,096."""
from __future__ import annotations

import numpy as np
import pytest
import torch

from oracle import focus_oracle as fo
from paper_2511_14694_gb300 import focus, inputs
from test_gpu_parity import bits

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    focus.device_status(clear=True)
    yield


def _layout(B, N, W, ks, seed):
    M = -(-N // W)
    k = inputs.k_schedule(M, ks, seed=seed)
    L = focus.layout_alloc(N, W, k, B=B)
    nt = inputs.nucleotides(B, N, seed=seed + 1, device="cuda")
    focus.layout_run(L, nt)
    return L


@pytest.mark.parametrize("B,N,W,ks,D", [(2, 3_001, 1_000, [100, 7], 64), (1, 777, 100, [30], 8),
                                        (3, 1_234, 256, [10, 50], 136), (1, 4_000, 1_000, [100], 4_096)])
def test_embed_matches_oracle_bit_exact(B, N, W, ks, D):
    L = _layout(B, N, W, ks, seed=D)
    table = inputs.normal_bf16((5, D), 1.0, seed=D + 7, device="cuda")
    out = focus.embed_tokens(L["tok"], table)
    torch.cuda.synchronize()
    assert focus.device_status(clear=True) == 0
    ref = fo.embed_tokens(L["tok"].cpu().numpy(), bits(table))
    assert np.array_equal(bits(out), ref)


def test_embed_out_of_table_token_is_reported_and_zeroed():
    tok = torch.tensor([[0, 4, 9, 3], [5, 1, 2, 255]], dtype=torch.uint8, device="cuda")
    table = inputs.normal_bf16((5, 32), 1.0, seed=3, device="cuda")
    out = focus.embed_tokens(tok, table)
    torch.cuda.synchronize()
    assert focus.device_status(clear=True) == 1  # FOCUS_ERR_INVALID_ARG
    ref = fo.embed_tokens(tok.cpu().numpy(), bits(table))
    assert np.array_equal(bits(out), ref)
    assert (bits(out)[0, 2] == 0).all() and (bits(out)[1, 3] == 0).all()


def test_embed_full_size_sampled():
    """The 128 kb layout (129,280 rows) at D = 4,096: 1.06 GB written; 2,000
    sampled rows and every summary row's count against the oracle's lookup."""
    L = _layout(1, 128_000, 1_000, [100], seed=42)
    D = 4_096
    table = inputs.normal_bf16((5, D), 1.0, seed=9, device="cuda")
    out = focus.embed_tokens(L["tok"], table)
    torch.cuda.synchronize()
    assert focus.device_status(clear=True) == 0
    tok = L["tok"].cpu().numpy()[0]
    rows = np.random.default_rng(1).choice(L["T"], 2_000, replace=False)
    got = bits(out[0, torch.from_numpy(rows).cuda()])
    assert np.array_equal(got, fo.embed_tokens(tok[rows], bits(table)))
    summ = (out[0] == table[focus.SUMMARY_TOKEN]).all(dim=1)
    assert int(summ.sum()) == L["T"] - 128_000 == 1_280
