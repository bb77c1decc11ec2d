"""Benchmark of the FOCUS compressed-context attention path on GB300.

Default workload: Evo-2-7B-shaped prefill, batch 1, N = 128,000 nt in 128
windows of W = 1,000 with a summary every k = 100 nt (1,280 retained
summaries), 32 heads, d = 128, bf16 Q/K/V ~ N(0,1)/sqrt(d). One step = the
whole prefill path over that input: focus_layout -> focus_kv_compact (bulk,
all windows) -> focus_attn_prefill (masked-parallel over all windows).
The decode leg times focus_attn_decode + focus_kv_compact on batch 64 with
10,000 retained summaries and partly filled windows per head (one leg = 256
decode steps).

Usage: python bench.py [--gpus N] [--steps K] [--warmup W] [--impl focus|reference]
For N > 1 launch with torch.distributed.run; each rank runs the same workload
on its own GPU (weak scaling, no collective on the data path).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

PEAKS_FALLBACK = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
NOMINAL_HBM_GBS = 7900.0
METRIC = "compressed-context prefill tokens/s and decode tokens/s at 1 GB300; % of roofline"


# ----------------------------------------------------------------------------- helpers

def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            d = json.load(f)
        return {k: float(d[k]) for k in ("hbm_gbs", "bf16_tflops", "bf16_tflops_sustained")}, "measured"
    except Exception:
        return dict(PEAKS_FALLBACK), "fallback"


def visible_pairs(win_off, ring_off):
    """Unmasked (query, key) pairs of the masked-parallel prefill: per window w,
    T_w (T_w + 1) / 2 causal pairs plus T_w * R_w ring pairs."""
    win_off = np.asarray(win_off, dtype=np.int64)
    ring_off = np.asarray(ring_off, dtype=np.int64)
    Tw = np.diff(win_off)
    Rw = ring_off[:-1]
    return int((Tw * (Tw + 1) // 2).sum() + (Tw * Rw).sum())


def kmer_local_row_counts(win_off, ring_off, k_sched):
    """Keys each row sees under the k-mer-local mask (Sec. 3.2): a row at
    in-window offset a of k-mer c = a // (k+1) sees a - c(k+1) + 1 rows of its
    k-mer, c earlier in-window FOCUS rows and the carried boundary when the
    previous window kept rows (a window with k = 0, or k >= T_w, is one k-mer)."""
    win_off = np.asarray(win_off, dtype=np.int64)
    ring_off = np.asarray(ring_off, dtype=np.int64)
    k_sched = np.asarray(k_sched, dtype=np.int64)
    rows = np.arange(win_off[-1])
    w = np.searchsorted(win_off, rows, side="right") - 1
    a = rows - win_off[w]
    Tw = np.diff(win_off)[w]
    kw = k_sched[w]
    kdiv = np.where((kw > 0) & (kw < Tw), kw, Tw) + 1
    c = a // kdiv
    bnd = ((w >= 1) & (ring_off[np.maximum(w - 1, 0)] < ring_off[w])).astype(np.int64)
    return a - c * kdiv + 1 + c + bnd


def decode_traffic(args):
    """Committed DRAM bytes per decode call for the batch-64 decode workload: the
    CUDA-core kernel at one query head per K/V head, the tensor-core kernel at
    eight (the two configurations with counters); None otherwise."""
    if args.decode_workload != "decode_1mb_b64_h32_d128" or args.rope:
        return None
    key = {1: "decode_split", 8: "decode_split_mma_g8"}.get(args.q_per_kv)
    return kernel_traffic(key, "paper_2511_14694_gb300/csrc/decode.cu") if key else None


def kernel_traffic(kernel_key: str, source: str):
    """DRAM bytes per launch from a committed ncu summary, only while the kernel
    source (and the prefill kernels' shared header) is unchanged since the
    counters were taken (else None)."""
    p = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(p) as f:
            d = json.load(f)[kernel_key]
        if d.get("source") != source:
            return None
        # the kernel's own source and the headers it shares with no other kernel
        for path, want in [(source, d.get("source_sha"))] + sorted(d.get("deps", {}).items()):
            with open(os.path.join(ROOT, path), "rb") as f:
                if hashlib.sha256(f.read()).hexdigest()[:16] != want:
                    return None
        return float(d["bytes_per_launch"])
    except Exception:
        return None


class ClockSampler:
    """nvidia-smi clocks and throttle reasons, sampled every 200 ms while running."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index, self.proc, self.lines = index, None, []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "200",
                 "-i", str(self.index)], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
            t0 = time.time()          # the timed region starts once sampling is live
            while not self.lines and time.time() - t0 < 3.0 and self.proc.poll() is None:
                time.sleep(0.02)
        except Exception:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *exc):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()
            self.t.join(timeout=2)
        return False

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.lines:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 7:
                continue
            try:
                sm.append(float(parts[0]))
                mx.append(float(parts[1]))
            except ValueError:
                continue
            for n, v in zip(names, parts[3:7]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


# ----------------------------------------------------------------------------- distributed

def dist_setup():
    """One process per GPU (torch.distributed.run sets RANK / LOCAL_RANK /
    WORLD_SIZE / MASTER_*). NCCL when CUDA is available, gloo otherwise; the
    process group carries only the timing barrier and the max over ranks."""
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch
        import torch.distributed as dist
        backend = os.environ.get("FOCUS_DIST_BACKEND") or ("nccl" if torch.cuda.is_available() else "gloo")
        if backend == "nccl":
            torch.cuda.set_device(local)
        dist.init_process_group(backend)
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x: float, world: int) -> float:
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def weak_scaling_value(units_per_rank: float, world: int, max_seconds: float) -> float:
    """Whole-job throughput: every rank processes its own units (no exchange), so
    the job's units are world x units_per_rank, over the slowest rank's time."""
    return world * units_per_rank / max_seconds


# ----------------------------------------------------------------------------- oracle (CPU baseline)

def oracle_head_times(cfg, L_host, k_sched, q, k, v, n_heads, mask="appendix"):
    """Times the fp64 oracle on whole heads of the workload: every window and
    every row of one (sequence, head) per pass, the sequential form of App. A.1
    for the appendix mask or every row under the k-mer-local mask of Sec. 3.2.
    Each (sequence, head) has the same visible pairs, so the whole workload takes
    B x H x the seconds of one pass. q/k/v hold a few heads' inputs, cycled (the
    timing does not depend on the values). Returns the per-pass seconds."""
    from oracle import focus_oracle as fo
    win_off = L_host["win_off"]
    scale = 1.0 / math.sqrt(cfg["d"])
    rows = None
    if mask == "kmer_local":
        rows = np.arange(int(win_off[-1]), dtype=np.int64)
    secs = []
    for i in range(n_heads):
        h = i % q.shape[0]
        t0 = time.perf_counter()
        if mask == "kmer_local":
            fo.attn_rows_kmer_local(q[h:h + 1], k[h:h + 1], v[h:h + 1], L_host["kind"], L_host["win"],
                                    L_host["kmer"], scale, np.zeros(rows.size, np.int64), rows)
        else:
            fo.prefill_sequential(q[h], k[h], v[h], win_off, L_host["keep"], scale)
        secs.append(time.perf_counter() - t0)
    return secs


def oracle_decode_times(host, fill0, R, W, Tw, n_steps, S, scale):
    """Times the fp64 oracle's decode (App. A.2) on the decode leg's first
    n_steps of S steps: every (sequence, K/V head) stream attends over its ring
    rows and window rows, whose counts follow the leg's own evolution (fill + 1
    per step; a full window of Tw rows retires its Tw - W FOCUS rows to the ring).
    host: uint16 bf16 bits of the cache (ring_k/ring_v [B, H, C_ring, d],
    win_k/win_v [B, H, C_win, d]) and of the steps' q, k_new, v_new ([S, B, H, d]).
    The oracle's time depends on the row counts only, so the cache contents the
    GPU leg left are used as they are. Returns the per-step seconds."""
    from oracle import focus_oracle as fo
    B, H, C_ring, d = host["ring_k"].shape
    C_win = host["win_k"].shape[2]
    rk, rv = host["ring_k"].reshape(B * H, C_ring, d), host["ring_v"].reshape(B * H, C_ring, d)
    wk, wv = host["win_k"].reshape(B * H, C_win, d), host["win_v"].reshape(B * H, C_win, d)
    fill = fill0.astype(np.int64).copy()
    Rb = np.full(B, R, np.int64)
    secs = []
    for s in range(min(n_steps, S)):
        q = host["q"][s].reshape(B * H, d)
        kn, vn = host["k"][s].reshape(B * H, d), host["v"][s].reshape(B * H, d)
        t0 = time.perf_counter()
        fo.decode(q, kn, vn, rk, rv, np.repeat(Rb, H), wk, wv, np.repeat(fill, H), scale)
        secs.append(time.perf_counter() - t0)
        fill += 1
        full = fill == Tw
        Rb[full] += Tw - W
        fill[full] = 0
    return secs


def oracle_stream_sample(win_off, ring_off, keep, pool_q, pool_k, pool_v, n_random, seed):
    """The fp64 oracle's sequential prefill (App. A.2) on a sample of the streaming
    workload: batch 0, every head, the rows of the last window and of n_random
    other windows (seeded), each head over the whole sequence (retention runs for
    every window; only the sampled windows' rows are computed). The sequence's
    rows are the leg's pool of windows repeated, as the GPU leg cycles it.
    Returns (seconds, sampled visible pairs, all visible pairs, windows sampled),
    pairs over the heads."""
    from oracle import focus_oracle as fo
    M = win_off.size - 1
    rng = np.random.default_rng(seed)
    pick = np.zeros(M, np.uint8)
    pick[M - 1] = 1
    pick[rng.choice(M - 1, size=min(n_random, M - 1), replace=False)] = 1
    tw = np.diff(win_off).astype(np.int64)
    pairs_w = tw * (tw + 1) // 2 + tw * ring_off[:-1].astype(np.int64)
    H, P_rows, d = pool_q.shape
    reps = -(-int(win_off[-1]) // P_rows)
    scale = 1.0 / math.sqrt(d)
    secs = 0.0
    for h in range(H):
        q, k, v = (np.tile(p[h], (reps, 1))[: int(win_off[-1])] for p in (pool_q, pool_k, pool_v))
        t0 = time.perf_counter()
        fo.prefill_sequential(q, k, v, win_off, keep, scale, want=pick)
        secs += time.perf_counter() - t0
    return secs, H * int(pairs_w[pick == 1].sum()), H * int(pairs_w.sum()), int(pick.sum())


def oracle_baseline(cfg, secs, mask):
    """(nt/s of the whole workload, description) from per-head oracle passes: the
    sum of the passes when all B x H of them ran (the workload timed in full),
    else B x H x the median pass."""
    per_head = statistics.median(secs)
    n_pass = cfg["B"] * cfg["H"]
    if len(secs) == n_pass:
        full_s = sum(secs)
        desc = ("fp64 oracle (%s), all %d (sequence, head) passes, every window and row: the workload timed in "
                "full, %.1f s (%.3f s per pass, median)" % ("k-mer-local rows" if mask == "kmer_local" else
                                                            "sequential prefill", n_pass, full_s, per_head))
        return cfg["B"] * cfg["N"] / full_s, desc, full_s
    full_s = per_head * n_pass
    desc = ("fp64 oracle (%s), %d whole (sequence, head) passes of %d, every window and row; %.3f s per pass "
            "(median); the workload's %d passes do the same visible pairs each, so its time is %d x that "
            "(extrapolated by passes)" % ("k-mer-local rows" if mask == "kmer_local" else "sequential prefill",
                                          len(secs), cfg["B"] * cfg["H"], per_head, cfg["B"] * cfg["H"],
                                          cfg["B"] * cfg["H"]))
    return cfg["B"] * cfg["N"] / full_s, desc, full_s


def workload_config(args, cfg, T, R, name=None, mask=None, rope=None, q_per_kv=None):
    """The config object of a bench line: the workload's shape, identical for the
    library arm and the reference (oracle) arm."""
    mask = args.mask if mask is None else mask
    rope = args.rope if rope is None else rope
    g = args.q_per_kv if q_per_kv is None else q_per_kv
    if cfg["mode"] == "stream":
        tw = T // max(1, -(-cfg["N"] // cfg["W"]))
        l2 = "inputs larger than L2 (pool of %d windows' Q/K/V %.2f GB, ring %.2f GB)" % (
            cfg["pool"], 3 * cfg["pool"] * cfg["B"] * cfg["H"] * tw * cfg["d"] * 2 / 1e9,
            2 * cfg["B"] * cfg["H"] * R * cfg["d"] * 2 / 1e9)
    else:
        l2 = "inputs larger than L2 (Q/K/V %.2f GB per step)" % (3 * cfg["B"] * T * cfg["H"] * cfg["d"] * 2 / 1e9)
    return {"workload": name or args.workload, "B": cfg["B"], "N": cfg["N"], "W": cfg["W"], "k": list(cfg["k"]),
            "H": cfg["H"], "d": cfg["d"], "T_augmented": int(T), "R_retained": int(R),
            "mask": "k-mer-local (Sec. 3.2)" if mask == "kmer_local" else "appendix (App. A, Eq. focus-attn)",
            "rope_theta": rope or None, "q_per_kv": g, "l2": l2}


# ----------------------------------------------------------------------------- focus arm

def run_prefill_leg(args, cfg, world, rank, local):
    import torch
    from paper_2511_14694_gb300 import focus, inputs, pipeline

    B, N, W, H, d = cfg["B"], cfg["N"], cfg["W"], cfg["H"], cfg["d"]
    M = focus.n_windows(N, W)
    k_s = inputs.k_schedule(M, cfg["k"], seed=inputs.DEFAULT_SEED)
    dev = torch.device("cuda", local)
    nt = inputs.nucleotides(B, N, seed=inputs.DEFAULT_SEED, device=dev)
    L = focus.layout_alloc(N, W, k_s, B=B, device=dev)
    g = args.q_per_kv
    q, k, v = inputs.qkv((B, H, L["T"], d), std=cfg["std"], seed=inputs.DEFAULT_SEED + rank, device=dev, q_per_kv=g)
    cache = focus.Cache(B, H // g, d, C_ring=max(L["R"], 1), device=dev, k_sched=k_s, rope_theta=args.rope,
                        q_per_kv=g)
    o = torch.empty_like(q)
    lse = torch.empty((B, H, L["T"]), dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)
    # device workspace the fastest kernel asks for (the rotary embedding's rotated q and k), allocated once
    ws = focus.new_prefill_workspace(cache, q, k, v, L, flags=args.prefill_flags)
    kernel_name = focus.prefill_kernel(cache, q, k, v, L, flags=args.prefill_flags, o=o, workspace=ws)

    def front(evc=None):
        focus.layout_run(L, nt, stream=stream)
        if evc is not None:
            evc[0].record(stream)
        focus.kv_compact_bulk(cache, k, v, L, 0, L["M"], src_row0=0, stream=stream)
        if evc is not None:
            evc[1].record(stream)

    def attn():
        focus.attn_prefill(cache, q, k, v, L, 0, L["M"], o=o, lse=lse, stream=stream, flags=args.prefill_flags,
                           workspace=ws)

    for _ in range(args.warmup):
        front()
        attn()
    torch.cuda.synchronize(dev)
    assert focus.device_status(clear=True) == 0
    win_off = L["win_off"].cpu().numpy()
    ring_off = L["ring_off"].cpu().numpy()
    local_mask = bool(args.prefill_flags & focus.PREFILL_KMER_LOCAL)
    pairs = (int(kmer_local_row_counts(win_off, ring_off, k_s).sum()) if local_mask
             else visible_pairs(win_off, ring_off))
    flops_per_step = 4.0 * d * H * B * pairs
    # algorithmic bytes of one prefill launch: read Q, K, V and write O once (bf16), write LSE (fp32)
    bytes_per_step = float(B * L["T"] * (H * (4 * d + 4) + (H // g) * 4 * d))

    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    evc = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    t_start, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier(world)
    torch.cuda.synchronize(dev)
    with ClockSampler(local) as clk:
        t_start.record(stream)
        for i in range(args.steps):
            front(evc[i])
            ev[i][0].record(stream)
            attn()
            ev[i][1].record(stream)
        t_end.record(stream)
        torch.cuda.synchronize(dev)
        # if the timed region was shorter than three sampling periods, keep the same
        # load running right after it until three samples exist
        extra = 0
        while len(clk.lines) < 3 and extra < 200 and not args.no_clock_wait:
            front()
            attn()
            extra += 1
            if extra % 20 == 0:
                torch.cuda.synchronize(dev)
        torch.cuda.synchronize(dev)
    barrier(world)
    assert focus.device_status(clear=True) == 0
    step_ms = t_start.elapsed_time(t_end) / args.steps
    step_ms = max_over_ranks(step_ms, world)
    attn_ms = sum(a.elapsed_time(b) for a, b in ev) / args.steps
    compact_ms = sum(a.elapsed_time(b) for a, b in evc) / args.steps
    # compaction moves R rows of K and V per K/V head: read once, written once
    compact_bytes = float(L["R"] * B * (H // g) * 2 * (2 * d) * 2)
    # layout scan + layout rows + bulk compaction + prefill (+ the rotary embedding's pass)
    launches = (4 + kernel_name.startswith("rotation pass")) * args.steps

    # end to end through the public API with host buffers: the pipelined host-buffer
    # prefill (copies of one head group overlap the kernels of the others)
    e2e = None
    if not args.no_e2e:
        steps_e2e = max(1, min(args.steps, 5))
        host = dict(nt=nt.cpu().pin_memory(), q=q.cpu().pin_memory(), k=k.cpu().pin_memory(),
                    v=v.cpu().pin_memory(), o=torch.empty(o.shape, dtype=o.dtype).pin_memory(),
                    lse=torch.empty(lse.shape, dtype=lse.dtype).pin_memory())
        devb = dict(nt=nt, q=q, k=k, v=v, o=o, lse=lse)
        h_nt, h_q, h_k, h_v, h_o, h_lse = (host[n] for n in ("nt", "q", "k", "v", "o", "lse"))

        def e2e_step():
            pipeline.prefill_masked_parallel_host(cache, L, host, devb, groups=args.e2e_groups,
                                                  flags=args.prefill_flags, stream=stream)

        # as many untimed steps as the headline's warm-up: on a fresh host the first
        # passes over the freshly pinned buffers run several times slower
        for _ in range(max(1, args.warmup)):
            e2e_step()
        torch.cuda.synchronize(dev)
        barrier(world)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(steps_e2e):
            e2e_step()
        e1.record(stream)
        torch.cuda.synchronize(dev)
        e2e_ms = max_over_ranks(e0.elapsed_time(e1) / steps_e2e, world)
        h2d = sum(x.numel() * x.element_size() for x in (h_nt, h_q, h_k, h_v))
        d2h = h_o.numel() * h_o.element_size() + h_lse.numel() * h_lse.element_size()
        e2e = {"value": world * B * N / (e2e_ms / 1e3), "unit": "nt/s", "ms_per_step": e2e_ms,
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "steps": steps_e2e,
               "api": "focus_prefill_host (C ABI, host buffers in and out; %d head groups, each group's "
                      "copies on two side streams overlapping the other groups' kernels)" % args.e2e_groups}
        del h_q, h_k, h_v, h_o, h_lse, host

    host_sample = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        # the heads' own inputs for up to --cpu-heads passes (at least two, cycled)
        nh = max(2, min(args.cpu_heads, q.shape[1]))
        host_sample = dict(win_off=win_off, ring_off=ring_off, kind=L["kind"].cpu().numpy(),
                           win=L["win"].cpu().numpy(), keep=L["keep"].cpu().numpy(), k_sched=k_s,
                           q=q[0, :nh].cpu(), k=k[0, :nh].cpu(), v=v[0, :nh].cpu())
    res = dict(kernel=kernel_name, attn_launches_per_step=1,
               step_desc="focus_layout + focus_kv_compact(bulk) + focus_attn_prefill(masked-parallel)",
               step_ms=step_ms, attn_ms=attn_ms, flops_per_step=flops_per_step, pairs=pairs, T=L["T"], R=L["R"],
               bytes_per_step=bytes_per_step, local_mask=local_mask, compact_ms=compact_ms,
               compact_bytes=compact_bytes,
               clocks=clk.summary(), launches=launches, e2e=e2e, host_sample=host_sample, extra_steps=extra)
    del q, k, v, o, lse, cache, ws
    torch.cuda.empty_cache()
    return res


def run_stream_leg(args, cfg, world, rank, local):
    """Streaming prefill (App. A.2): for each window in order, focus_kv_compact of
    that window; the attention per chunk of args.stream_chunk windows (one
    focus_attn_prefill over the chunk against the ring), consecutive chunks'
    attention overlapping on two streams (pipeline.prefill_streaming). The Q/K/V
    come from a seeded pool of windows (cycled), held as pool / chunk contiguous
    chunk tensors."""
    import torch
    from paper_2511_14694_gb300 import focus, inputs, pipeline

    B, N, W, H, d, P = cfg["B"], cfg["N"], cfg["W"], cfg["H"], cfg["d"], cfg["pool"]
    C = args.stream_chunk
    if C < 1:
        raise ValueError("--stream-chunk must be >= 1")
    P = -(-max(P, C) // C) * C        # the pool holds whole chunks, at least the workload's pool
    M = focus.n_windows(N, W)
    k_s = inputs.k_schedule(M, cfg["k"], seed=inputs.DEFAULT_SEED)
    dev = torch.device("cuda", local)
    L = focus.layout(N, W, k_s, device=dev)
    off = L["win_off_host"]
    Tw = int(np.diff(off).max())
    if not (np.diff(off) == Tw).all():
        raise ValueError("the streaming leg expects windows of equal augmented size")
    g = args.q_per_kv
    n_slots = P // C                  # chunk tensors in the pool, each [B, H(, /g), C Tw, d]
    seed = inputs.DEFAULT_SEED + rank
    pq = [inputs.normal_bf16((B, H, C * Tw, d), cfg["std"], seed=3 * seed + 1 + 10 * j, device=dev)
          for j in range(n_slots)]
    pk = [inputs.normal_bf16((B, H // g, C * Tw, d), cfg["std"], seed=3 * seed + 2 + 10 * j, device=dev)
          for j in range(n_slots)]
    pv = [inputs.normal_bf16((B, H // g, C * Tw, d), cfg["std"], seed=3 * seed + 3 + 10 * j, device=dev)
          for j in range(n_slots)]
    cache = focus.Cache(B, H // g, d, C_ring=max(L["R"], 1), device=dev, k_sched=k_s, rope_theta=args.rope,
                        q_per_kv=g)
    local_mask = bool(args.prefill_flags & focus.PREFILL_KMER_LOCAL)
    outs = [torch.empty((B, H, C * Tw, d), dtype=torch.bfloat16, device=dev) for _ in range(2)]
    lses = [torch.empty((B, H, C * Tw), dtype=torch.float32, device=dev) for _ in range(2)]
    stream = torch.cuda.current_stream(dev)
    n_calls = -(-M // C)
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n_calls)]
    kernel_name = focus.prefill_kernel(cache, pq[0], pk[0], pv[0], L, M - C, M, flags=args.prefill_flags, o=outs[0])

    def span(w0, w1=None):
        j = (w0 // C) % n_slots
        return pq[j], pk[j], pv[j]

    cevs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(M)]

    def step(timed=False):
        # each window's compaction, then the attention per chunk on one of two side
        # streams: consecutive chunks' launches overlap (pipeline.prefill_streaming)
        pipeline.prefill_streaming(cache, L, span, outs, lses, flags=args.prefill_flags, stream=stream,
                                   events=evs if timed else None, compact_events=cevs if timed else None, chunk=C)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize(dev)
    assert focus.device_status(clear=True) == 0
    pairs = (int(kmer_local_row_counts(off, L["ring_off_host"], k_s).sum()) if local_mask
             else visible_pairs(off, L["ring_off_host"]))
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    attn_ms = compact_ms = 0.0
    use_graph = not args.no_stream_graph
    if use_graph:
        # the per-call split (attention launches, in-step compactions) from one eager
        # step with events; the timed steps replay the step captured as one CUDA graph
        step(timed=True)
        torch.cuda.synchronize(dev)
        attn_ms = sum(a.elapsed_time(b) for a, b in evs) * args.steps
        compact_ms = sum(a.elapsed_time(b) for a, b in cevs) * args.steps
        graph = pipeline.StreamingGraph(cache, L, span, outs, lses, flags=args.prefill_flags, chunk=C)
        for _ in range(max(1, args.warmup)):
            graph.replay()
        torch.cuda.synchronize(dev)
        assert focus.device_status(clear=True) == 0
    barrier(world)
    with ClockSampler(local) as clk:
        t0.record(stream)
        for _ in range(args.steps):
            if use_graph:
                graph.replay()
                continue
            step(timed=True)
            torch.cuda.synchronize(dev)
            attn_ms += sum(a.elapsed_time(b) for a, b in evs)
            compact_ms += sum(a.elapsed_time(b) for a, b in cevs)
        t1.record(stream)
        torch.cuda.synchronize(dev)
    barrier(world)
    # the window compaction alone (nothing else running): re-copies windows' kept
    # rows to the ring slots they already hold
    n_alone = min(M, 100)
    aev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n_alone)]
    for w, (a, b) in enumerate(aev):
        _, ck, cv = span(w - w % C)
        a.record(stream)
        focus.kv_compact_bulk(cache, ck, cv, L, w, w + 1, src_row0=int(off[w - w % C]), stream=stream)
        b.record(stream)
    torch.cuda.synchronize(dev)
    alone_ms = statistics.median(a.elapsed_time(b) for a, b in aev)
    assert focus.device_status(clear=True) == 0
    step_ms = max_over_ranks(t0.elapsed_time(t1) / args.steps, world)
    # the attention launches overlap, so the rate is taken over the whole step
    # (compactions and gaps included); per_launch_ms is each launch on its stream
    cpu = None
    if rank == 0 and world == 1 and args.stream_cpu_windows > 0 and not local_mask and not args.rope and g == 1:
        bits = lambda t: t[0].contiguous().view(torch.int16).cpu().numpy().view(np.uint16)  # noqa: E731
        # the pool as the leg cycles it: window w is pool window w mod P
        pool = [np.concatenate([bits(t[j]) for j in range(n_slots)], axis=1) for t in (pq, pk, pv)]
        secs, sp, ap_, nw = oracle_stream_sample(np.asarray(off), np.asarray(L["ring_off_host"]),
                                                 L["keep"].cpu().numpy(), pool[0], pool[1], pool[2],
                                                 args.stream_cpu_windows, inputs.DEFAULT_SEED)
        full_s = secs * ap_ / sp * B               # every sequence has the same windows and pairs
        cpu = {"value": B * N / full_s, "unit": "nt/s", "cores": os.cpu_count(), "kind": "oracle",
               "sample": "fp64 oracle (sequential prefill with retention), batch 0, all %d heads, the rows of %d "
                         "windows (the last and %d seeded others) of %d: %.1f s for %.3g of the %.3g visible "
                         "pairs per sequence; the workload's time is that per pair x all pairs x %d sequences "
                         "(extrapolated)" % (H, nw, nw - 1, M, secs, sp, ap_, B)}
        del pool
    # per-window compaction: the window's kept rows of every (sequence, K/V head), read and written
    wc_ms = compact_ms / args.steps / M
    wc_bytes = float((L["R"] / M) * B * (H // g) * 2 * (2 * d) * 2)
    return dict(kernel=kernel_name, attn_launches_per_step=n_calls,
                step_desc=("per window: focus_kv_compact(window); per chunk of %d windows: focus_attn_prefill(chunk) "
                           "(the masked-parallel form over the chunk), consecutive chunks' attention overlapping on "
                           "two streams; all windows; rate over the whole step%s" %
                           (C, "; the step captured once as a CUDA graph (pipeline.StreamingGraph) and replayed, "
                               "per-launch figures from one eager step" if use_graph else "")),
                stream_chunk=C,
                window_compaction={"kernel": "focus_kv_compact (one window)", "bytes_per_launch": wc_bytes,
                                   "in_step_ms": wc_ms,
                                   "in_step_note": "CUDA events on the main stream inside the step: includes "
                                                   "waiting for SMs held by the overlapping attention launches",
                                   "alone_ms": alone_ms, "alone_GBps": wc_bytes / (alone_ms / 1e3) / 1e9,
                                   "alone_note": "median of %d launches with nothing else running: a ~1 MB "
                                                 "launch, launch-latency bound" % n_alone},
                step_ms=step_ms, attn_ms=step_ms, flops_per_step=4.0 * d * H * B * pairs, pairs=pairs,
                T=L["T"], R=L["R"], clocks=clk.summary(), launches=(M + n_calls * (1 + kernel_name.startswith("rotation pass"))) * args.steps, e2e=None, host_sample=None,
                cpu_baseline=cpu,
                per_launch_ms=attn_ms / args.steps / n_calls, local_mask=local_mask,
                bytes_per_step=float(B * L["T"] * (H * (4 * d + 4) + (H // g) * 4 * d)))


def run_embed_leg(args, world, rank, local):
    """focus_embed_tokens on the 128 kb layout's token stream (129,280 rows) at an
    Evo-2-7B-like width D: T x D bf16 written once, T token bytes read. CUDA events
    around each launch; the output (1.06 GB at D = 4,096) exceeds L2."""
    import torch
    from paper_2511_14694_gb300 import focus, inputs
    from paper_2511_14694_gb300.workloads import WORKLOADS
    cfg = WORKLOADS["prefill_128kb_h32_d128"]
    N, W, D = cfg["N"], cfg["W"], args.embed_d
    M = focus.n_windows(N, W)
    k_s = inputs.k_schedule(M, cfg["k"], seed=inputs.DEFAULT_SEED)
    dev = torch.device("cuda", local)
    nt = inputs.nucleotides(1, N, seed=inputs.DEFAULT_SEED + rank, device=dev)
    L = focus.layout_alloc(N, W, k_s, B=1, device=dev)
    focus.layout_run(L, nt)
    table = inputs.normal_bf16((5, D), 1.0, seed=inputs.DEFAULT_SEED, device=dev)
    out = torch.empty((1, L["T"], D), dtype=torch.bfloat16, device=dev)
    stream = torch.cuda.current_stream(dev)
    for _ in range(3):
        focus.embed_tokens(L["tok"], table, out=out, stream=stream)
    reps = 10
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(reps)]
    torch.cuda.synchronize(dev)
    for a, b in ev:
        a.record(stream)
        focus.embed_tokens(L["tok"], table, out=out, stream=stream)
        b.record(stream)
    torch.cuda.synchronize(dev)
    assert focus.device_status(clear=True) == 0
    ms = sorted(a.elapsed_time(b) for a, b in ev)[reps // 2]
    nbytes = float(L["T"] * D * 2 + L["T"] + 5 * D * 2)
    del out
    return dict(ms=ms, bytes=nbytes, T=L["T"], D=D)


def run_decode_leg(args, cfg, world, rank, local):
    import torch
    from paper_2511_14694_gb300 import focus, inputs

    B, H, d, W, R = cfg["B"], cfg["H"], cfg["d"], cfg["W"], cfg["R"]
    g = args.q_per_kv
    Hk = H // g                      # K/V heads; H query heads
    kk = cfg["k"][0]
    Tw = W + -(-W // kk)
    S = cfg["steps"]
    dev = torch.device("cuda", local)
    k_sched = np.full(R // (W // kk) + S // W + 16, kk, np.int32)
    cache = focus.Cache(B, Hk, d, C_ring=R + 256, C_win=1_024, W=W, k_sched=k_sched, device=dev, rope_theta=args.rope,
                        q_per_kv=g)
    for i, t in enumerate((cache.ring_k, cache.ring_v, cache.win_k, cache.win_v)):
        t.copy_(inputs.normal_bf16(t.shape, cfg["std"], seed=50 + i + 10 * rank, device=dev))
    fill0 = inputs.start_fill(B, Tw - 1, seed=inputs.DEFAULT_SEED)
    widx0 = R // (W // kk)
    qs = inputs.normal_bf16((S, B, H, d), cfg["std"], seed=300 + rank, device=dev)
    ks_, vs = (inputs.normal_bf16((S, B, Hk, d), cfg["std"], seed=400 + 2 * rank + i, device=dev) for i in (0, 1))
    o = torch.empty((B, H, d), dtype=torch.bfloat16, device=dev)
    lse = torch.empty((B, H), dtype=torch.float32, device=dev)
    ws = cache.new_workspace()
    stream = torch.cuda.current_stream(dev)

    def reset():
        cache.ring_len.fill_(R)
        cache.win_idx.fill_(widx0)
        cache.win_fill.copy_(torch.from_numpy(fill0).to(dev))

    def leg(evs=None):
        for s in range(S):
            if evs is not None:
                evs[s][0].record(stream)
            focus.attn_decode(cache, qs[s], ks_[s], vs[s], o=o, lse=lse, workspace=ws, stream=stream)
            if evs is not None:
                evs[s][1].record(stream)
            focus.kv_compact_window(cache, stream=stream)

    reps = max(1, args.decode_reps)
    reset()
    leg()
    torch.cuda.synchronize(dev)
    assert focus.device_status(clear=True) == 0
    # bytes the decode reads/writes per leg (host simulation of the fill/ring evolution)
    fill = fill0.astype(np.int64).copy()
    Rb = np.full(B, R, np.int64)
    bytes_leg = 0
    for _ in range(S):
        # K/V rows of ring + window once per K/V head; q read, o written (and lse) per query
        # head; k_new, v_new read and appended per K/V head
        bytes_leg += int((Hk * ((Rb + fill) * 2 * d * 2 + 4 * d * 2) + H * (2 * d * 2 + 4)).sum())
        fill += 1
        full = fill == Tw
        Rb[full] += Tw - W
        fill[full] = 0
    evs = [[(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(S)]
           for _ in range(reps)]
    times = []
    barrier(world)
    with ClockSampler(local) as clk:
        for r in range(reps):
            reset()
            torch.cuda.synchronize(dev)
            t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            t0.record(stream)
            leg(evs[r])
            t1.record(stream)
            torch.cuda.synchronize(dev)
            times.append(t0.elapsed_time(t1))
    barrier(world)
    assert focus.device_status(clear=True) == 0
    leg_ms = max_over_ranks(sum(times) / reps, world)
    dec_ms = sum(a.elapsed_time(b) for rr in evs for a, b in rr) / reps
    cpu = None
    if rank == 0 and world == 1 and args.decode_cpu_steps > 0 and not args.rope and g == 1:
        bits = lambda t: t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)  # noqa: E731
        host = dict(ring_k=bits(cache.ring_k), ring_v=bits(cache.ring_v), win_k=bits(cache.win_k),
                    win_v=bits(cache.win_v), q=bits(qs), k=bits(ks_), v=bits(vs))
        secs = oracle_decode_times(host, fill0, R, W, Tw, args.decode_cpu_steps, S, 1.0 / math.sqrt(d))
        total = sum(secs) * (S / len(secs))
        full = len(secs) == S
        cpu = {"value": B * S / total, "unit": "tokens/s", "cores": os.cpu_count(), "kind": "oracle",
               "sample": ("fp64 oracle decode (every stream over its ring and window rows), %s of the leg's %d "
                          "steps (B=%d x H=%d streams each), %.2f s per step (mean)%s" %
                          ("all" if full else "the first %d" % len(secs), S, B, H, sum(secs) / len(secs),
                           "" if full else "; the leg's time is %d x the mean step (extrapolated by steps)" % S))}
        del host
    return dict(leg_ms=leg_ms, decode_kernels_ms=dec_ms, bytes_leg=bytes_leg, steps=S, B=B,
                clocks=clk.summary(), launches=3 * S * reps, cpu_baseline=cpu)


def prefill_roofline(pre, peaks, peaks_src, traffic=None):
    """Roofline object of a prefill leg's attention kernel: visible-pair FLOPs
    (appendix mask) or bytes (k-mer-local mask, a few keys per row) per launch
    over the average launch time."""
    n_launch = pre["attn_launches_per_step"]
    achieved = pre["flops_per_step"] / (pre["attn_ms"] / 1e3) / 1e12
    common = {"traffic": traffic, "visible_pairs": pre["pairs"], "avg_launch_ms": pre.get("per_launch_ms",
                                                                                         pre["attn_ms"]),
              "launches_per_step": n_launch, "flop_per_launch": pre["flops_per_step"] / n_launch,
              "prefill_kernel": pre["kernel"]}
    if pre["local_mask"]:
        gbs = pre["bytes_per_step"] / (pre["attn_ms"] / 1e3) / 1e9
        r = {"bound": "hbm", "achieved": gbs, "peak": peaks["hbm_gbs"], "unit": "GB/s", "frac": gbs / peaks["hbm_gbs"],
             "peak_source": f"{peaks_src} copy bandwidth", "kernel": "prefill attention (k-mer-local)",
             "tflops": achieved, "bytes_per_launch": pre["bytes_per_step"] / n_launch}
    else:
        r = {"bound": "tensor", "achieved": achieved, "peak": peaks["bf16_tflops"], "unit": "TFLOP/s",
             "frac": achieved / peaks["bf16_tflops"], "peak_source": f"{peaks_src} bf16 dense burst",
             "frac_of_sustained": achieved / peaks["bf16_tflops_sustained"], "kernel": "prefill attention"}
    r.update(common)
    if pre["kernel"].startswith("rotation pass"):
        # the rotary embedding's pass runs inside each timed call, before the attention
        r["kernel"] += " with the rotation pass before it (both launches in the timed call)"
    return r


# the other named workloads and options timed beside the headline:
# (key, workload, steps, warm-up, options: mask, rotary base)
CONFIG_LEGS = [("ksweep", "prefill_256kb_ksweep_h32_d128", 10, 3, {"cpu_heads": 1}),
               ("causal", "causal_128kb_h32_d128", 3, 3, {}),
               ("stream", "stream_1mb_b4_h32_d128", 2, 3, {}),
               ("kmer_local", "prefill_128kb_h32_d128", 20, 3, {"mask": "kmer_local"}),
               ("rope", "prefill_128kb_h32_d128", 20, 3, {"rope": 500000.0}),
               ("stream_kmer_local", "stream_1mb_b4_h32_d128", 2, 3, {"mask": "kmer_local"})]


def run_config_leg(args, name, steps, warmup, world, rank, local, peaks, peaks_src, opts=None):
    """One of the other named workloads, at the default options (appendix mask,
    no rotary embedding, one query head per K/V head) unless ``opts`` sets the
    mask or the rotary base, timed like the headline step; returns its object for
    the bench line."""
    import copy
    from paper_2511_14694_gb300.workloads import WORKLOADS
    cfg = WORKLOADS[name]
    opts = opts or {}
    a = copy.copy(args)
    a.steps, a.warmup, a.no_e2e = steps, warmup, True
    # an oracle sample for the legs that ask for one (whole (sequence, head) passes)
    a.cpu_heads = int(opts.get("cpu_heads", 0)) if opts else 0
    a.no_cpu_baseline = a.cpu_heads == 0 or args.no_cpu_baseline
    a.rope, a.q_per_kv, a.mask = float(opts.get("rope", 0.0)), 1, opts.get("mask", "appendix")
    a.prefill_flags = 2 if a.mask == "kmer_local" else 0
    pre = (run_stream_leg if cfg["mode"] == "stream" else run_prefill_leg)(a, cfg, world, rank, local)
    obj = {"workload": name, "value": weak_scaling_value(cfg["B"] * cfg["N"], world, pre["step_ms"] / 1e3),
           "unit": "nt/s", "ms_per_step": pre["step_ms"], "steps": steps, "warmup": warmup,
           "augmented_tokens_per_s": world * cfg["B"] * pre["T"] / (pre["step_ms"] / 1e3),
           "step": pre["step_desc"], "config": workload_config(a, cfg, pre["T"], pre["R"], name=name),
           "roofline": prefill_roofline(pre, peaks, peaks_src, leg_traffic(pre, a, cfg)), "clocks": pre["clocks"],
           "gpu_launches": pre["launches"]}
    if pre.get("window_compaction") is not None:
        obj["window_compaction"] = pre["window_compaction"]
    if pre.get("cpu_baseline") is not None:
        obj["cpu_baseline"] = pre["cpu_baseline"]
    if pre.get("host_sample") is not None:
        hs = pre["host_sample"]
        secs = oracle_head_times(cfg, hs, hs["k_sched"], hs["q"], hs["k"], hs["v"], a.cpu_heads, mask=a.mask)
        val, desc, _ = oracle_baseline(cfg, secs, a.mask)
        obj["cpu_baseline"] = {"value": val, "unit": "nt/s", "cores": os.cpu_count(), "kind": "oracle",
                               "sample": desc}
    return obj


def leg_traffic(pre, args, cfg):
    """DRAM bytes per launch from the committed ncu counters, which exist for the
    128 kb workload (default heads) on the appendix-mask persistent kernel, the
    rotary embedding's pass with that kernel after it (the two launches of one
    call) and the k-mer-tiled kernel; None elsewhere or once a kernel's source has
    changed since the capture."""
    from paper_2511_14694_gb300.workloads import WORKLOADS
    key = {("tcgen05 persistent", False, False): ("prefill_attention", "prefill_tc_persistent.cu"),
           ("rotation pass + tcgen05 persistent", False, True): ("prefill_attention_rope", "rope.cu"),
           ("tcgen05 k-mer tiles", True, False): ("prefill_attention_kmer_local", "prefill_tc_kmer.cu"),
           }.get((pre["kernel"], pre.get("local_mask", False), bool(args.rope)))
    if not key or args.q_per_kv != 1 or cfg is not WORKLOADS["prefill_128kb_h32_d128"]:
        return None
    return kernel_traffic(key[0], "paper_2511_14694_gb300/csrc/" + key[1])


def run_compact_leg(args, world, rank, local, peaks, peaks_src):
    """Bulk focus_kv_compact at the 1 Mb x 4 workload's size: the FOCUS rows of
    all 1,000 windows (10,000 per (sequence, head), 128 (sequence, head) pairs)
    gathered from the augmented K/V (B=4, H=32, T=1,010,000, d=128) into the
    ring: 655 MB read and 655 MB written per launch, both above L2. The source
    values are never read as numbers (a bit copy), so it is left uninitialised."""
    import torch
    from paper_2511_14694_gb300 import focus
    from paper_2511_14694_gb300.workloads import WORKLOADS
    cfg = WORKLOADS["stream_1mb_b4_h32_d128"]
    B, N, W, H, d = cfg["B"], cfg["N"], cfg["W"], cfg["H"], cfg["d"]
    dev = torch.device("cuda", local)
    L = focus.layout(N, W, list(cfg["k"]), device=dev)
    src_k = torch.empty((B, H, L["T"], d), dtype=torch.bfloat16, device=dev)
    src_v = torch.empty_like(src_k)
    cache = focus.Cache(B, H, d, C_ring=L["R"], device=dev)
    stream = torch.cuda.current_stream(dev)
    for _ in range(3):
        focus.kv_compact_bulk(cache, src_k, src_v, L, 0, L["M"], stream=stream)
    reps = 10
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(reps)]
    torch.cuda.synchronize(dev)
    for e0, e1 in ev:
        e0.record(stream)
        focus.kv_compact_bulk(cache, src_k, src_v, L, 0, L["M"], stream=stream)
        e1.record(stream)
    torch.cuda.synchronize(dev)
    assert focus.device_status(clear=True) == 0
    ms = statistics.median(a.elapsed_time(b) for a, b in ev)
    nbytes = float(L["R"] * B * H * 2 * (2 * d) * 2)
    gbs = nbytes / (ms / 1e3) / 1e9
    del src_k, src_v, cache
    torch.cuda.empty_cache()
    return {"kernel": "focus_kv_compact (bulk)", "workload": "ring of stream_1mb_b4_h32_d128 (R = %d rows per "
            "(sequence, head), B = %d, H = %d, d = %d)" % (L["R"], B, H, d), "avg_launch_ms": ms,
            "bytes_per_launch": nbytes, "launches": reps,
            "timing": "CUDA events around each of %d launches (median); source rows and ring above L2" % reps,
            "roofline": {"bound": "hbm", "achieved": gbs, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                         "frac": gbs / peaks["hbm_gbs"], "peak_source": f"{peaks_src} copy bandwidth"}}


def run_focus(args, world, rank, local):
    import torch
    from paper_2511_14694_gb300.workloads import WORKLOADS
    torch.cuda.set_device(local)
    peaks, peaks_src = load_peaks()
    cfg = WORKLOADS[args.workload]
    if args.no_prefill:          # decode leg alone (profiling runs)
        dec = run_decode_leg(args, WORKLOADS[args.decode_workload], world, rank, local)
        if rank == 0:
            print(json.dumps({"decode_workload": args.decode_workload, "leg_ms": dec["leg_ms"],
                              "decode_call_ms": dec["decode_kernels_ms"] / dec["steps"],
                              "GBps": dec["bytes_leg"] / (dec["decode_kernels_ms"] / 1e3) / 1e9}), flush=True)
        return
    if cfg["mode"] == "stream":
        pre = run_stream_leg(args, cfg, world, rank, local)
    else:
        pre = run_prefill_leg(args, cfg, world, rank, local)
    dec = None
    if not args.no_decode:
        dec = run_decode_leg(args, WORKLOADS[args.decode_workload], world, rank, local)
    emb = None if args.embed_d <= 0 else run_embed_leg(args, world, rank, local)
    legs = {}
    if not args.no_configs:
        for key, name, steps, warmup, opts in CONFIG_LEGS:
            if name != args.workload or opts.get("mask", "appendix") != args.mask or \
                    float(opts.get("rope", 0.0)) != float(args.rope):
                legs[key] = run_config_leg(args, name, steps, warmup, world, rank, local, peaks, peaks_src, opts)
    big_compact = None if args.no_configs else run_compact_leg(args, world, rank, local, peaks, peaks_src)
    if rank != 0:
        return
    value = weak_scaling_value(cfg["B"] * cfg["N"], world, pre["step_ms"] / 1e3)
    traffic = leg_traffic(pre, args, cfg)
    line = {
        "metric": METRIC,
        "value": value, "unit": "nt/s", "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": pre["step_ms"], "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16", "data": "synthetic (seeded N(0,1)/sqrt(d) bf16 Q/K/V, uniform A/C/G/T ids)",
        "config": workload_config(args, cfg, pre["T"], pre["R"]),
        "step": pre["step_desc"],
        "augmented_tokens_per_s": world * cfg["B"] * pre["T"] / (pre["step_ms"] / 1e3),
        "roofline": prefill_roofline(pre, peaks, peaks_src, traffic),
        "clocks": pre["clocks"],
        "e2e": pre["e2e"],
        "gpu_launches": pre["launches"],
    }
    if "compact_ms" in pre:
        cgbs = pre["compact_bytes"] / (pre["compact_ms"] / 1e3) / 1e9
        line["compaction"] = {"kernel": "focus_kv_compact (bulk)", "avg_launch_ms": pre["compact_ms"],
                              "timing": "CUDA events around the compaction inside each timed step (after the "
                                        "previous step's prefill); a ~10 us launch, so the launch gap counts",
                              "bytes_per_launch": pre["compact_bytes"],
                              "roofline": {"bound": "hbm", "achieved": cgbs, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                                           "frac": cgbs / peaks["hbm_gbs"],
                                           "peak_source": f"{peaks_src} copy bandwidth"}}
    if big_compact is not None:
        line["compaction_1mb_ring"] = big_compact
    if emb is not None:
        egbs = emb["bytes"] / (emb["ms"] / 1e3) / 1e9
        line["embedding"] = {"kernel": "focus_embed_tokens", "rows": emb["T"], "D": emb["D"],
                             "avg_launch_ms": emb["ms"], "bytes_per_launch": emb["bytes"],
                             "timing": "CUDA events around each of 10 launches (median); output larger than L2",
                             "roofline": {"bound": "hbm", "achieved": egbs, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                                          "frac": egbs / peaks["hbm_gbs"],
                                          "peak_source": f"{peaks_src} copy bandwidth"}}
    if dec is not None:
        gbs = dec["bytes_leg"] / (dec["decode_kernels_ms"] / 1e3) / 1e9
        line["decode"] = {
            "workload": args.decode_workload, "value": world * dec["B"] * dec["steps"] / (dec["leg_ms"] / 1e3),
            "unit": "tokens/s", "ms_per_step": dec["leg_ms"] / dec["steps"],
            "step": "focus_attn_decode + focus_kv_compact(window)",
            "roofline": {"bound": "hbm", "achieved": gbs, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                         "frac": gbs / peaks["hbm_gbs"], "frac_of_nominal": gbs / NOMINAL_HBM_GBS,
                         "peak_source": f"{peaks_src} copy bandwidth", "bytes_per_step": dec["bytes_leg"] / dec["steps"],
                         "avg_decode_call_ms": dec["decode_kernels_ms"] / dec["steps"],
                         "traffic": decode_traffic(args)},
            "clocks": dec["clocks"],
        }
        line["decode"]["gpu_launches"] = dec["launches"]
        if dec.get("cpu_baseline") is not None:
            line["decode"]["cpu_baseline"] = dec["cpu_baseline"]
    line.update(legs)
    if pre.get("cpu_baseline") is not None:          # a stream workload's oracle sample
        line["cpu_baseline"] = pre["cpu_baseline"]
    if pre["host_sample"] is not None and (args.rope or args.q_per_kv > 1):
        line["cpu_baseline"] = None      # the oracle baseline times the default path only
    elif pre["host_sample"] is not None:
        hs = pre["host_sample"]
        if pre.get("local_mask", False):
            from oracle import focus_oracle as fo
            hs["kmer"] = fo.layout_kmer(cfg["N"], cfg["W"], hs["k_sched"])
        secs = oracle_head_times(cfg, hs, hs["k_sched"], hs["q"], hs["k"], hs["v"], args.cpu_heads,
                                 mask=args.mask)
        val, desc, _ = oracle_baseline(cfg, secs, args.mask)
        line["cpu_baseline"] = {"value": val, "unit": "nt/s", "cores": os.cpu_count(), "kind": "oracle",
                                "sample": desc}
    print(json.dumps(line), flush=True)


# ----------------------------------------------------------------------------- reference arm (the oracle)

def run_reference(args, world, rank, local):
    """The fp64 CPU oracle timed on the host cores, on the same workload, metric,
    unit and config as the library arm: each step is one whole (sequence, head)
    pass (every window and row), the workload's time that pass times B x H (every
    pass does the same visible pairs), the same sampler as the library arm's
    cpu_baseline."""
    if rank != 0:
        return
    from oracle import focus_oracle as fo
    from paper_2511_14694_gb300 import inputs
    from paper_2511_14694_gb300.workloads import WORKLOADS
    cfg = WORKLOADS[args.workload]
    if cfg["mode"] == "stream":
        print(json.dumps({"impl": "reference", "unavailable": "the reference arm times the masked-parallel "
                          "workloads only"}), flush=True)
        return
    B, N, W, H, d = cfg["B"], cfg["N"], cfg["W"], cfg["H"], cfg["d"]
    M = fo.n_windows(N, W)
    k_s = inputs.k_schedule(M, cfg["k"], seed=inputs.DEFAULT_SEED)
    L = fo.layout(N, W, k_s)
    # two heads of inputs, drawn with the same generator recipe on the CPU
    q, k, v = inputs.qkv((2, L["T"], d), std=cfg["std"], seed=inputs.DEFAULT_SEED, device="cpu")
    hs = dict(win_off=L["win_off"], ring_off=L["ring_off"], keep=L["keep"], kind=L["kind"], win=L["win"])
    if args.mask == "kmer_local":
        hs["kmer"] = fo.layout_kmer(N, W, k_s)
    oracle_head_times(cfg, hs, k_s, q, k, v, args.warmup, mask=args.mask)
    secs = oracle_head_times(cfg, hs, k_s, q, k, v, args.steps, mask=args.mask)
    value, desc, full_s = oracle_baseline(cfg, secs, args.mask)
    per_pass = statistics.median(secs)
    line = {"metric": METRIC, "value": value, "unit": "nt/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": per_pass * 1e3, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic", "impl": "reference",
            "config": workload_config(args, cfg, int(L["win_off"][-1]), int(L["ring_off"][-1])),
            "step": "one whole (sequence, head) pass of the oracle: 1/%d of the workload; value = B N / "
                    "(%d x ms_per_step)" % (B * H, B * H),
            "workload_s": full_s,
            "cpu_baseline": {"value": value, "unit": "nt/s", "cores": os.cpu_count(), "kind": "oracle",
                             "sample": desc},
            "e2e": {"value": value, "unit": "nt/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def run_memory_report(args, world, rank, local):
    """Memory scaling with context length (the paper's Fig. "Scalability of memory
    with context length", Sec. 4.5): peak device memory and time of a streaming
    FOCUS prefill (one window's Q/K/V resident at a time, the retained ring
    growing as N/k), of the masked-parallel FOCUS prefill (all rows resident, one
    launch) and of a full-cache causal prefill over the same N (Q/K/V of all N
    rows resident), one attention layer, batch 1, 32 heads, d = 128. Each time is
    the second of two passes."""
    if rank != 0:
        return
    import torch
    from paper_2511_14694_gb300 import focus, inputs, pipeline
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    H, d, W, k = 32, 128, 1_000, 100

    def timed(fn):
        fn()                                               # warm-up pass, not timed
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize(dev)
        e0.record()
        fn()
        e1.record()
        torch.cuda.synchronize(dev)
        assert focus.device_status(clear=True) == 0
        return e0.elapsed_time(e1)

    for N in [int(x) for x in args.memory_ns.split(",")]:
        row = {"report": "memory_scaling", "N": N, "H": H, "d": d, "W": W, "k": k,
               "kv_bytes_full": 2 * N * H * d * 2}
        # FOCUS streaming: ring (retained summaries) + one window of Q/K/V/O at a time
        torch.cuda.synchronize(dev)
        torch.cuda.empty_cache()
        torch.cuda.reset_peak_memory_stats(dev)
        base = torch.cuda.memory_allocated(dev)
        L = focus.layout(N, W, [k], device=dev)
        off = L["win_off_host"]
        Tw = int(np.diff(off).max())
        row["kv_bytes_focus"] = 2 * (L["R"] + Tw) * H * d * 2
        cache = focus.Cache(1, H, d, C_ring=max(L["R"], 1), device=dev)
        q, kk, v = inputs.qkv((1, H, Tw, d), std=1 / math.sqrt(d), seed=1, device=dev)
        o = torch.empty_like(q)
        lse = torch.empty((1, H, Tw), dtype=torch.float32, device=dev)
        def stream():
            for w in range(L["M"]):
                a, e = int(off[w]), int(off[w + 1])
                n = e - a
                cut = (lambda t: t[:, :, :n].contiguous()) if n != Tw else (lambda t: t)
                focus.attn_prefill(cache, cut(q), cut(kk), cut(v), L, w, w + 1, o=cut(o), lse=cut(lse))
                focus.kv_compact_bulk(cache, cut(kk), cut(v), L, w, w + 1, src_row0=a)

        row["focus_eager_ms"] = timed(stream)
        # the same per-window loop captured once as a CUDA graph: one launch per
        # pass instead of two host calls per window
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            stream()
        row["focus_ms"] = timed(graph.replay)
        row["focus_mode"] = "per-window loop (attention, then compaction) replayed as a CUDA graph"
        row["focus_peak_bytes"] = torch.cuda.max_memory_allocated(dev) - base
        del graph
        del cache, q, kk, v, o, lse
        # FOCUS masked-parallel: Q/K/V of all rows resident, bulk compaction + one launch
        torch.cuda.synchronize(dev)
        torch.cuda.empty_cache()
        torch.cuda.reset_peak_memory_stats(dev)
        base = torch.cuda.memory_allocated(dev)
        cache = focus.Cache(1, H, d, C_ring=max(L["R"], 1), device=dev)
        q, kk, v = inputs.qkv((1, H, L["T"], d), std=1 / math.sqrt(d), seed=1, device=dev)
        o = torch.empty_like(q)
        lse = torch.empty((1, H, L["T"]), dtype=torch.float32, device=dev)
        row["focus_parallel_ms"] = timed(lambda: pipeline.prefill_masked_parallel(cache, q, kk, v, L, o=o, lse=lse))
        row["focus_parallel_peak_bytes"] = torch.cuda.max_memory_allocated(dev) - base
        row["focus_parallel_kernel"] = focus.prefill_kernel(cache, q, kk, v, L)
        del cache, q, kk, v, o, lse, L
        # full cache: plain causal attention over all N rows (k = 0, one window)
        if N <= args.memory_full_max:
            torch.cuda.synchronize(dev)
            torch.cuda.empty_cache()
            torch.cuda.reset_peak_memory_stats(dev)
            base = torch.cuda.memory_allocated(dev)
            Lc = focus.layout(N, N, [0], device=dev)
            cc = focus.Cache(1, H, d, C_ring=0, device=dev)
            q, kk, v = inputs.qkv((1, H, N, d), std=1 / math.sqrt(d), seed=1, device=dev)
            o = torch.empty_like(q)
            lse = torch.empty((1, H, N), dtype=torch.float32, device=dev)
            row["full_ms"] = timed(lambda: focus.attn_prefill(cc, q, kk, v, Lc, o=o, lse=lse))
            row["full_peak_bytes"] = torch.cuda.max_memory_allocated(dev) - base
            del cc, q, kk, v, o, lse, Lc
        print(json.dumps(row), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="focus", choices=["focus", "reference"])
    ap.add_argument("--workload", default="prefill_128kb_h32_d128")
    ap.add_argument("--decode-reps", type=int, default=2)
    ap.add_argument("--no-decode", action="store_true")
    ap.add_argument("--no-prefill", action="store_true", help="run only the decode leg (profiling)")
    ap.add_argument("--decode-workload", default="decode_1mb_b64_h32_d128")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--embed-d", type=int, default=4096,
                    help="width of the token-embedding gather timed beside the step (0 = skip)")
    ap.add_argument("--e2e-groups", type=int, default=16,
                    help="head (or sequence) groups of the pipelined host-buffer prefill timed as e2e")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-heads", type=int, default=8,
                    help="whole (sequence, head) oracle passes timed for the cpu_baseline (8 of 32 = 25%%)")
    ap.add_argument("--decode-cpu-steps", type=int, default=8,
                    help="decode steps the fp64 oracle runs for the decode leg's cpu_baseline (0 = none; the leg's "
                         "256 = in full)")
    ap.add_argument("--stream-cpu-windows", type=int, default=8,
                    help="stream legs (appendix mask): windows besides the last on which the fp64 oracle runs for "
                         "the leg's cpu_baseline (0 = none)")
    ap.add_argument("--no-stream-graph", action="store_true",
                    help="stream legs: enqueue every step from the host instead of replaying its CUDA graph")
    ap.add_argument("--stream-chunk", type=int, default=8,
                    help="windows per attention call in the streaming legs (divides the pool of 8; 1 = per window)")
    ap.add_argument("--no-configs", action="store_true",
                    help="skip the other named workloads and the 1 Mb ring compaction (profiling runs)")
    ap.add_argument("--no-clock-wait", action="store_true",
                    help="do not extend the load after a short timed region (profiling runs)")
    ap.add_argument("--legacy", action="store_true", help="time the legacy mma.sync prefill kernel")
    ap.add_argument("--rope", type=float, default=0.0,
                    help="rotary-embedding base (0 = none): q and k are rotated at their position ids")
    ap.add_argument("--q-per-kv", type=int, default=1,
                    help="grouped-query heads: the workload's H query heads share H / G K/V heads")
    ap.add_argument("--mask", default="appendix", choices=["appendix", "kmer_local"],
                    help="prefill visibility: App. A (default) or the k-mer-local rule of Sec. 3.2")
    ap.add_argument("--memory-report", action="store_true",
                    help="peak memory and time vs context length, FOCUS streaming vs full-cache causal")
    ap.add_argument("--memory-ns", default="16000,32000,64000,128000,256000,512000,1000000")
    ap.add_argument("--memory-full-max", type=int, default=256_000)
    args = ap.parse_args()
    args.warmup = max(3, args.warmup)
    args.prefill_flags = (1 if args.legacy else 0) | (2 if args.mask == "kmer_local" else 0)
    if args.q_per_kv < 1:
        ap.error("--q-per-kv must be >= 1")
    world, rank, local = dist_setup()
    if args.memory_report:
        run_memory_report(args, world, rank, local)
    elif args.impl == "reference":
        run_reference(args, world, rank, local)
    else:
        run_focus(args, world, rank, local)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
