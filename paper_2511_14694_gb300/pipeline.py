"""The two prefill modes of App. A.1 ("Cross-window consistency") as
sequences of C-ABI calls. No arithmetic happens here; each step is a kernel.

- masked-parallel: bulk-compact every window's FOCUS K/V into the ring, then one
  prefill call over all windows (window w reads ring prefix ring_off[w]);
- sequential (streaming, App. A.2): for each window, prefill it against the ring,
  then compact its FOCUS K/V into the ring.

Under the k-mer-local mask (``focus.PREFILL_KMER_LOCAL``, Sec. 3.2) a row also
reads its own window's FOCUS rows from the ring, so the streaming step compacts
the window before its prefill (a copy of K/V rows, which are inputs of the
step, so the order changes no value).
"""
from __future__ import annotations

from . import focus


def prefill_masked_parallel(cache: focus.Cache, q, k, v, L: dict, scale=None, o=None, lse=None, flags=0,
                            stream=None):
    focus.kv_compact_bulk(cache, k, v, L, 0, L["M"], src_row0=0, stream=stream)
    return focus.attn_prefill(cache, q, k, v, L, 0, L["M"], scale=scale, o=o, lse=lse, flags=flags, stream=stream)


def prefill_window(cache: focus.Cache, q_w, k_w, v_w, L: dict, w: int, scale=None, o=None, lse=None, flags=0,
                   stream=None):
    """One streaming step: window w's rows (q_w/k_w/v_w: [B, H, T_w, d]) attend to
    the ring and to themselves, then window w's FOCUS rows join the ring."""
    row0 = int(L["win_off_host"][w])
    local = bool(flags & focus.PREFILL_KMER_LOCAL)
    if local:
        focus.kv_compact_bulk(cache, k_w, v_w, L, w, w + 1, src_row0=row0, stream=stream)
    out = focus.attn_prefill(cache, q_w, k_w, v_w, L, w, w + 1, scale=scale, o=o, lse=lse, flags=flags,
                             stream=stream)
    if not local:
        focus.kv_compact_bulk(cache, k_w, v_w, L, w, w + 1, src_row0=row0, stream=stream)
    return out
