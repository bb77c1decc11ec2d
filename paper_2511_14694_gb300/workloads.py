"""Named synthetic workloads shaped like the paper's (Evo-2-7B-like heads,
1 kb windows, ~100x compression; Sec. 4.1 and Table "Full configuration").

Plain data: shapes and value distributions, no arithmetic of the method.
"""
from __future__ import annotations

import math

WORKLOADS = {
    # single layer, 4 windows of 1 kb, k=100, small heads: the parity case
    "prefill_4kb_h4_d64": dict(mode="prefill", B=1, N=4_000, W=1_000, k=(100,), H=4, d=64, std=1.0),
    # Evo-2-7B-shaped prefill: 128 windows of 1 kb, k=100 -> 1,280 retained summaries
    "prefill_128kb_h32_d128": dict(mode="prefill", B=1, N=128_000, W=1_000, k=(100,), H=32, d=128,
                                   std=1.0 / math.sqrt(128)),
    # decode against the compressed cache of a 1 Mb context: 10,000 retained summaries
    # plus up to 1,010 current-window rows per head, batch 64, 256 steps
    "decode_1mb_b64_h32_d128": dict(mode="decode", B=64, R=10_000, W=1_000, k=(100,), H=32, d=128,
                                    steps=256, std=1.0),
    # the same cache shape at batch 8, for profiler captures (about 1.5 GB resident)
    "decode_1mb_b8_h32_d128": dict(mode="decode", B=8, R=10_000, W=1_000, k=(100,), H=32, d=128,
                                   steps=256, std=1.0),
    # randomized compression schedule: k per window from {10, 25, 50, 100, 200}
    "prefill_256kb_ksweep_h32_d128": dict(mode="prefill", B=1, N=256_000, W=1_000,
                                          k=(10, 25, 50, 100, 200), H=32, d=128,
                                          std=1.0 / math.sqrt(128)),
    # ultra-long streaming prefill with per-window compaction
    "stream_1mb_b4_h32_d128": dict(mode="stream", B=4, N=1_000_000, W=1_000, k=(100,), H=32, d=128,
                                   std=1.0 / math.sqrt(128), pool=8),
    # a smaller prefill of the same shape (32 windows) for profiler captures: inputs still exceed L2
    "prefill_32kb_h32_d128": dict(mode="prefill", B=1, N=32_000, W=1_000, k=(100,), H=32, d=128,
                                  std=1.0 / math.sqrt(128)),
    # plain causal attention at 16 kb (long work items, inputs above L2) for profiler captures
    "causal_16kb_h32_d128": dict(mode="prefill", B=1, N=16_000, W=16_000, k=(0,), H=32, d=128,
                                 std=1.0 / math.sqrt(128)),
    # plain causal attention (no compression) at 128 kb, for the O(N^2) comparison
    "causal_128kb_h32_d128": dict(mode="prefill", B=1, N=128_000, W=128_000, k=(0,), H=32, d=128,
                                  std=1.0 / math.sqrt(128)),
}
