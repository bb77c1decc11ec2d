"""The two prefill modes of App. A.1 ("Cross-window consistency") as
sequences of C-ABI calls. No arithmetic happens here; each step is a kernel.

- masked-parallel: bulk-compact every window's FOCUS K/V into the ring, then one
  prefill call over all windows (window w reads ring prefix ring_off[w]);
- sequential (streaming, App. A.2): for each window, prefill it against the ring,
  then compact its FOCUS K/V into the ring;
- masked-parallel from and to pinned host memory: the same calls per group of
  heads (or sequences), with the host-device copies of one group on side
  streams overlapping the kernels of the others;
- streaming with overlapping windows: each window's compaction first, then its
  attention on one of two side streams, so consecutive windows' launches overlap;
  optionally several windows per attention call; captured once as a CUDA graph
  and replayed (StreamingGraph).

Under the k-mer-local mask (``focus.PREFILL_KMER_LOCAL``, Sec. 3.2) a row also
reads its own window's FOCUS rows from the ring, so the streaming step compacts
the window before its prefill (a copy of K/V rows, which are inputs of the
step, so the order changes no value).
"""
from __future__ import annotations

import torch

from . import focus


def prefill_masked_parallel(cache: focus.Cache, q, k, v, L: dict, scale=None, o=None, lse=None, flags=0,
                            stream=None, workspace="auto"):
    focus.kv_compact_bulk(cache, k, v, L, 0, L["M"], src_row0=0, stream=stream)
    return focus.attn_prefill(cache, q, k, v, L, 0, L["M"], scale=scale, o=o, lse=lse, flags=flags, stream=stream,
                              workspace=workspace)


_side_streams: dict = {}


def prefill_masked_parallel_host(cache: focus.Cache, L: dict, host: dict, dev: dict, groups: int = 8, scale=None,
                                 flags=0, stream=None, workspace="auto"):
    """Masked-parallel prefill of a layer whose inputs and outputs live in pinned
    host memory, through the library's focus_prefill_host: host["nt"] (uint8
    [B, N]), host["q"/"k"/"v"] (bf16 [B, H, T, d]) in, host["o"] (bf16) and
    host["lse"] (fp32 [B, H, T]) out; ``dev`` holds device tensors of the same
    shapes, reused across calls.

    The layout runs once; then the K/V heads (one sequence) or the sequences go
    in ``groups`` parts, and part i's Q/K/V copy in on one side stream, its
    compaction and attention run on ``stream``, and its O/LSE copy out on a second
    side stream, so that the copies of one part overlap the compute and copies
    of the others. Work is only enqueued: when ``stream`` is done, so is
    everything, outputs in host memory included."""
    cur = stream if stream is not None else torch.cuda.current_stream()
    key = cur.device
    if key not in _side_streams:
        _side_streams[key] = (torch.cuda.Stream(device=key), torch.cuda.Stream(device=key))
    s_in, s_out = _side_streams[key]
    return focus.prefill_host(cache, L, host, dev, s_in, s_out, groups=groups, scale=scale, flags=flags,
                              workspace=workspace, stream=cur)


def prefill_streaming(cache: focus.Cache, L: dict, window_qkv, outs, lses, w_begin: int = 0, w_end: int | None = None,
                      scale=None, flags=0, stream=None, events=None, compact_events=None, chunk: int = 1,
                      workspaces=None):
    """Streaming prefill (App. A.2) of windows [w_begin, w_end) with the
    attention of consecutive windows (or chunks of windows) overlapping.

    ``chunk`` = 1: window_qkv(w) gives window w's (q, k, v) ([B, H, T_w, d] each)
    and window w writes outs[i] and lses[i], i = w % len(outs) (two buffers
    suffice; one per window keeps every output). ``chunk`` = c > 1: the windows go
    in chunks of c, window_qkv(w0, w1) gives the rows of windows [w0, w1)
    ([B, H, win_off[w1] - win_off[w0], d]) and chunk n writes outs[n % len(outs)].

    Each window's FOCUS rows are compacted into the ring, window by window in
    order on ``stream``, before the attention that reads them (a copy of input
    rows: window w reads ring rows [0, ring_off[w]) only, so the order changes no
    value). One attention call then covers the window (or the chunk: the
    masked-parallel form of App. A.1 over the chunk's windows, the same rows as
    one call per window). It needs only the compactions before it, not the
    previous attention: it runs on side stream i % 2, so the tail of one launch
    overlaps the start of the next (launches that share a buffer share a stream,
    so a buffer is never written by two launches at once). Larger chunks mean
    fewer, fuller launches and c windows' inputs resident at once.
    ``events``: optional list of (start, end) CUDA events per attention call,
    recorded around it on its stream; ``compact_events`` the same per window
    around each compaction on ``stream``. ``workspaces``: optional pair of
    attention workspaces, one per side stream (each of the largest call's
    prefill_workspace_bytes); by default each call allocates its own. Work is
    only enqueued; when ``stream`` is done, so is everything."""
    if chunk < 1:
        raise ValueError("chunk must be >= 1")
    cur = stream if stream is not None else torch.cuda.current_stream()
    key = cur.device
    if key not in _side_streams:
        _side_streams[key] = (torch.cuda.Stream(device=key), torch.cuda.Stream(device=key))
    side = _side_streams[key]
    w_end = L["M"] if w_end is None else w_end
    off = L["win_off_host"]
    for s_ in side:
        s_.wait_stream(cur)                    # inputs and buffers written before the call
    for n, w0 in enumerate(range(w_begin, w_end, chunk)):
        w1 = min(w0 + chunk, w_end)
        q, k, v = window_qkv(w0) if chunk == 1 else window_qkv(w0, w1)
        for w in range(w0, w1):
            if compact_events is not None:
                compact_events[w - w_begin][0].record(cur)
            focus.kv_compact_bulk(cache, k, v, L, w, w + 1, src_row0=int(off[w0]), stream=cur)
            if compact_events is not None:
                compact_events[w - w_begin][1].record(cur)
        i = (w0 if chunk == 1 else n) % len(outs)
        s_ = side[i % 2]
        s_.wait_stream(cur)                    # ring rows of windows < w1 are in place
        for t in (q, k, v):
            # window_qkv may return tensors made for this call: keep the caching
            # allocator from reusing them before the launch on s_ has read them
            t.record_stream(s_)
        if events is not None:
            events[n][0].record(s_)
        if workspaces is None:
            # allocated on this stream's behalf: the caching allocator must not hand
            # the block to another call before this launch on s_ is done with it
            ws = focus.new_prefill_workspace(cache, q, k, v, L, w0, w1, flags)
            if ws is not None:
                ws.record_stream(s_)
        else:
            ws = workspaces[i % 2]
        focus.attn_prefill(cache, q, k, v, L, w0, w1, scale=scale, o=outs[i], lse=lses[i], flags=flags, stream=s_,
                           workspace=ws)
        if events is not None:
            events[n][1].record(s_)
    for s_ in side:
        cur.wait_stream(s_)
    return outs, lses


class StreamingGraph:
    """prefill_streaming over windows [w_begin, w_end) captured once as a CUDA
    graph and replayed: one graph launch instead of one host call per
    compaction and attention (about 1,100 per 1 Mb x 4 step at chunks of 8), so
    the step no longer waits on the host to enqueue it.

    The graph holds the addresses it was captured with: window_qkv's tensors, the
    outputs, the cache and the layout. A caller streams new windows by copying
    them into those tensors before a replay. Construction runs the step once
    eagerly (the library's one-time set-up: the device status word, the driver's
    tensor-map entry point, the kernels' attributes) and allocates one attention
    workspace per side stream, so nothing is allocated inside the capture."""

    def __init__(self, cache: focus.Cache, L: dict, window_qkv, outs, lses, w_begin: int = 0,
                 w_end: int | None = None, scale=None, flags=0, chunk: int = 1):
        w_end = L["M"] if w_end is None else w_end
        need = 0
        for w0 in range(w_begin, w_end, chunk):
            w1 = min(w0 + chunk, w_end)
            q, k, v = window_qkv(w0) if chunk == 1 else window_qkv(w0, w1)
            need = max(need, focus.prefill_workspace_bytes(cache, q, k, v, L, w0, w1, flags))
        dev = outs[0].device
        self.workspaces = ([torch.empty(need, dtype=torch.uint8, device=dev) for _ in range(2)] if need
                           else [None, None])
        args = (cache, L, window_qkv, outs, lses, w_begin, w_end, scale, flags)
        prefill_streaming(*args, chunk=chunk, workspaces=self.workspaces)
        torch.cuda.synchronize(dev)
        self.graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(self.graph):
            prefill_streaming(*args, stream=torch.cuda.current_stream(), chunk=chunk, workspaces=self.workspaces)
        torch.cuda.synchronize(dev)

    def replay(self):
        """Enqueue the whole step on the current stream."""
        self.graph.replay()


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
