"""FOCUS oracle: plain fp64 CPU statement of the paper's layout, masked
attention, KV retention and decode (arXiv 2511.14694, App. A).

TEST INFRASTRUCTURE ONLY. Only ``tests/``, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline leg may import it; the CUDA library never does.
"""
from . import focus_oracle  # noqa: F401
