/*
 * focus.h — C ABI of the GB300 FOCUS compressed-context attention library
 * (libfocus.so). FOCUS: arXiv 2511.14694.
 *
 * What the library computes
 *   A DNA sequence of N bases is cut into windows of W bases (App. A, I_w and
 *   M = ceil(N/W)). Inside each window a FOCUS summary token is inserted after
 *   every k_w bases, and after the partial k-mer that ends a window
 *   (B_w = ceil(|I_w|/k_w), App. A; Sec. 3.2 "Setup and tokens"). Each inserted
 *   token takes a position of its own in the sequence. Row i of window w attends to
 *   (a) the retained FOCUS K/V of all earlier windows and (b) the rows of
 *   window w up to and including itself (Eq. focus-attn's visible set and the
 *   context C(t) of App. A.1). After window w only its FOCUS K/V is kept
 *   (App. A, "KV compression and budget"; App. A.2 streaming inference),
 *   optionally with a boundary tail: the window's last `tail` ordinary rows
 *   (App. A allows a short boundary tail besides them). Kept rows form the
 *   ring that every later window attends to.
 *
 * Conventions for every entry point
 *   - Ownership: the caller allocates and owns every buffer. Pointers named
 *     d_* or documented as "device" are CUDA device pointers; "host" pointers
 *     are ordinary host memory. The library never allocates device memory.
 *   - Layouts are row-major with the head dimension d fastest. K/V/Q/O are
 *     bf16 (raw 16-bit storage, passed as void*). All device pointers to bf16
 *     tensors must be 16-byte aligned.
 *   - Calls are asynchronous on the given stream (0 = legacy default stream)
 *     unless stated otherwise. The return value reports argument errors found
 *     on the host (nothing is launched then) and CUDA launch errors.
 *   - Errors found by a kernel (a window buffer or ring overflowing, layout
 *     sizes that disagree with the caller's) set a sticky per-device status
 *     word; the affected work is skipped, never trapped. Read and clear it with
 *     focus_get_device_status().
 *   - Supported head dimensions: d = 64 and d = 128.
 *   - CUDA graphs: focus_layout, focus_kv_compact, focus_attn_prefill,
 *     focus_attn_decode(_noalloc) and focus_embed_tokens enqueue kernels on the
 *     given stream only, allocate nothing and never synchronize, so they can be
 *     captured (stream capture) and the graph replayed. A graph keeps the
 *     pointers it was captured with; the cache's lengths live in device memory,
 *     so replays of a decode step advance them. Make each call once outside the
 *     capture first: the first call per device sets up the status word, the
 *     driver's tensor-map entry point and the kernels' attributes.
 *     focus_get_device_status synchronizes and cannot be captured.
 */
#ifndef FOCUS_H_
#define FOCUS_H_

#include <stddef.h>
#include <stdint.h>
#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum focus_status {
    FOCUS_OK = 0,
    FOCUS_ERR_INVALID_ARG = 1,   /* null pointer, negative size, inconsistent shapes */
    FOCUS_ERR_UNSUPPORTED = 2,   /* head dim not 64/128, misaligned pointer */
    FOCUS_ERR_CAPACITY = 3,      /* ring or window buffer too small (host check or device word) */
    FOCUS_ERR_CUDA = 4,          /* a CUDA call failed */
    FOCUS_ERR_TIMEOUT = 5,       /* a bounded device wait gave up (device word only) */
    FOCUS_ERR_LAYOUT = 6         /* device-computed layout disagrees with the caller's sizes */
} focus_status;

/* Summary token id written into the token stream (the reserved special token of
 * Table "Full configuration"); nucleotide ids are 0..3 for A, C, G, T. */
#define FOCUS_SUMMARY_TOKEN 4

/* Layout flag: also close the partial k-mer at the end of the LAST window with a
 * summary (App. A's ceil). Without it, the final partial k-mer stays open, which is
 * what a caller that will continue the sequence by decoding wants. */
#define FOCUS_LAYOUT_CLOSE_TAIL 1u

/* ------------------------------------------------------------------------ */
/* Library information                                                      */
/* ------------------------------------------------------------------------ */

/* Version of this ABI (major*10000 + minor*100 + patch). */
int32_t focus_version(void);

/* Human-readable name of a status code (static string, never NULL). */
const char* focus_status_string(focus_status s);

/* Read the calling thread's current device's sticky status word into
 * *host_status (FOCUS_OK if no kernel reported an error) and, if clear != 0,
 * reset it to FOCUS_OK. Synchronises `stream` first (blocking). */
focus_status focus_get_device_status(int32_t* host_status, int32_t clear, cudaStream_t stream);

/* ------------------------------------------------------------------------ */
/* focus_layout — summary-token insertion and position ids                  */
/* Sec. 3.2 "Setup and tokens"; App. A (I_w, M, B_w; a FOCUS token has a     */
/* position of its own); Sec. 3.3 (augmented sequence y_1..y_N').           */
/* ------------------------------------------------------------------------ */

/* Host-only arithmetic: the number of windows M that cover n_nt >= 0 bases with
 * windows of W >= 1 bases, M = ceil(n_nt / W) (App. A); 0 for n_nt = 0.
 * FOCUS_ERR_INVALID_ARG for a negative n_nt, W < 1, a NULL M or an M above INT32_MAX. */
focus_status focus_layout_windows(int64_t n_nt, int32_t W, int32_t* M);

/* Adaptive windowing (see focus_layout_size_sched): of a window-length schedule
 * h_W[0..n_sched) (HOST), the number M of leading windows whose lengths first
 * reach n_nt bases in total, i.e. the windows that cover the sequence (the last
 * one may be only partly used); 0 for n_nt = 0. FOCUS_ERR_INVALID_ARG if a length
 * among them is < 1, if all n_sched lengths cover fewer than n_nt bases, or for
 * NULL pointers. */
focus_status focus_layout_windows_sched(int64_t n_nt, int32_t n_sched, const int32_t* h_W, int32_t* M);

/* Host-only arithmetic: sizes of the augmented layout.
 *   n_nt        N >= 0 bases
 *   W           window length in bases, W >= 1
 *   n_windows   M; must equal ceil(N/W)
 *   h_k         HOST array [M]: cadence k_w >= 0 per window (0 = no summaries)
 *   flags       FOCUS_LAYOUT_CLOSE_TAIL or 0
 *   tail        boundary tail: ordinary rows kept at the end of each window (>= 0; 0 = none)
 * Outputs (any may be NULL): *T augmented length N + sum_w B_w, *R kept rows
 * (sum_w B_w + min(tail, n_w)), *max_rows the largest per-window augmented row count. */
focus_status focus_layout_size(int64_t n_nt, int32_t W, int32_t n_windows, const int32_t* h_k,
                               uint32_t flags, int32_t tail, int64_t* T, int64_t* R, int32_t* max_rows);

/* Device arrays written by focus_layout. All are caller-allocated. */
typedef struct focus_layout_out {
    int64_t  T;          /* capacity/expected augmented length (from focus_layout_size) */
    int64_t  R;          /* expected number of kept rows (from focus_layout_size) */
    uint8_t* kind;       /* [T] 0 = base, 1 = FOCUS summary */
    int32_t* src;        /* [T] nucleotide index; a summary names the last base of its k-mer */
    int32_t* pos;        /* [T] position id (0-based augmented index) */
    int32_t* win;        /* [T] window id */
    uint8_t* tok;        /* [B][T] token ids (nt id 0..3, summary FOCUS_SUMMARY_TOKEN); may be NULL */
    uint8_t* keep;       /* [T] 1 if KV retention keeps the row (summary or boundary-tail base); may be NULL */
    int32_t* win_off;    /* [M+1] first augmented row of each window; win_off[M] = T */
    int32_t* ring_off;   /* [M+1] kept rows before each window; ring_off[M] = R */
    int32_t* sum_idx;    /* [R] augmented index of each kept row, in order (the compaction gather list) */
    int32_t* base_off;   /* [M+1] first base of each window; base_off[M] = N. May be NULL for
                            focus_layout; required by focus_layout_sched */
} focus_layout_out;

/* Device layout builder. d_k: DEVICE array [M] of cadences (same values as the
 * host array given to focus_layout_size). d_nt: DEVICE uint8 [B][N] nucleotide ids
 * (may be NULL, then tok is not written). If the device-computed T or R differs
 * from out->T / out->R the device status word is set to FOCUS_ERR_LAYOUT.
 * N = 0 (M = 0) is valid: it only writes win_off[0] = ring_off[0] = 0. */
focus_status focus_layout(int64_t n_nt, int32_t W, int32_t n_windows, const int32_t* d_k,
                          uint32_t flags, int32_t tail, int32_t B, const uint8_t* d_nt,
                          const focus_layout_out* out, cudaStream_t stream);

/* Adaptive windowing (Sec. 5: W and k chosen per region): window w covers the
 * next W_sched[w] bases, the last window whatever is left. The n_windows
 * lengths must all be > 0 and cover exactly n_nt bases (the last window
 * non-empty); otherwise FOCUS_ERR_INVALID_ARG (host) or FOCUS_ERR_INVALID_ARG in
 * the device status word. h_W is a HOST array, d_W the DEVICE copy of the same
 * values; everything else is as in focus_layout_size / focus_layout, which are
 * the case W_sched[w] = W. */
focus_status focus_layout_size_sched(int64_t n_nt, int32_t n_windows, const int32_t* h_W, const int32_t* h_k,
                                     uint32_t flags, int32_t tail, int64_t* T, int64_t* R, int32_t* max_rows);
focus_status focus_layout_sched(int64_t n_nt, int32_t n_windows, const int32_t* d_W, const int32_t* d_k,
                                uint32_t flags, int32_t tail, int32_t B, const uint8_t* d_nt,
                                const focus_layout_out* out, cudaStream_t stream);

/* ------------------------------------------------------------------------ */
/* Compressed KV cache (caller-owned). App. A.2 "Streaming with controlled   */
/* memory": a per-(sequence, head) contiguous ring of retained FOCUS K/V     */
/* plus the current window's K/V buffer.                                   */
/* ------------------------------------------------------------------------ */
typedef struct focus_cache {
    void*    ring_k;          /* device bf16 [B][H][C_ring][d] retained FOCUS keys */
    void*    ring_v;          /* device bf16 [B][H][C_ring][d] retained FOCUS values */
    void*    win_k;           /* device bf16 [B][H][C_win][d] current-window keys (decode) */
    void*    win_v;           /* device bf16 [B][H][C_win][d] current-window values (decode) */
    int32_t* ring_len;        /* device [B] retained rows R_b */
    int32_t* win_fill;        /* device [B] rows in the current window buffer */
    int32_t* win_idx;         /* device [B] index of the current window (selects k_w) */
    const int32_t* k_per_window; /* device [n_windows] cadence schedule */
    int32_t  n_windows;
    int32_t  W;               /* window length in bases */
    int32_t  B, H, d;
    int32_t  C_ring, C_win;   /* capacities in rows */
    int32_t  tail;            /* boundary tail kept by window-mode compaction (>= 0) */
    int32_t* pos_base;        /* device [B] position id of the current window's first row, or NULL;
                                 window-mode compaction adds the retired window's T_w to it */
    float    rope_theta;      /* rotary-embedding base; 0 = none (see below) */
    const int32_t* W_per_window; /* device [n_windows] window lengths (adaptive windowing), or NULL: W */
    int32_t  q_per_kv;        /* query heads per K/V head (grouped-query heads); 0 or 1 = one each */
} focus_cache;

/* Grouped-query heads (q_per_kv = g > 1; not in the paper): H counts K/V heads.
 * Keys, values, the ring and the window buffer have H heads; queries, outputs
 * and LSE have H * g heads, and query head hq uses K/V head hq / g. The cache
 * and its K/V traffic shrink by g. Decode serves up to four query heads of a
 * group per K/V pass. The legacy prefill kernel refuses g > 1
 * (FOCUS_ERR_UNSUPPORTED); g must be <= 64 (FOCUS_ERR_INVALID_ARG). */

/* Rotary position embedding at the layout's position ids (RoFormer; the paper
 * gives each FOCUS token a position of its own, Sec. 3.2, and names no base).
 * With rope_theta > 0 every query and key the library receives is rotated before
 * use: for i < d/2 the pair (x_i, x_{i+d/2}) turns by the angle p * theta_i,
 * theta_i = rope_theta^(-2i/d), p = the row's position id (its global augmented
 * index). Keys enter the cache rotated: focus_kv_compact in bulk mode rotates the
 * rows it copies (p = sum_idx entry), focus_attn_decode appends the rotated new
 * key (p = pos_base[b] + win_fill[b], so pos_base is required), and window-mode
 * compaction copies already rotated rows. focus_attn_prefill rotates q and the
 * current windows' k (p = win_off[w] + in-window row) and reads the ring as
 * stored. Angles are reduced modulo 2 pi in fp64 before the fp32 sine and cosine;
 * rotated values are rounded to bf16 before they are used. rope_theta must be
 * finite and >= 0 (FOCUS_ERR_INVALID_ARG otherwise). */

/* ------------------------------------------------------------------------ */
/* focus_attn_prefill — windowed attention over the compressed context      */
/* Eq. focus-attn with visible set I_w-past ∪ retained FOCUS KV; App. A.1    */
/* "Cross-window consistency" (sequential or masked-parallel); App. A.2.    */
/* ------------------------------------------------------------------------ */
typedef struct focus_prefill_args {
    const void* q;            /* device bf16 [B][H][T_span][d] rows of windows [w_begin, w_end) */
    const void* k;            /* device bf16 [B][H][T_span][d] */
    const void* v;            /* device bf16 [B][H][T_span][d] */
    void*       o;            /* device bf16 [B][H][T_span][d] output */
    float*      lse;          /* device fp32 [B][H][T_span] natural-log sum-exp of scaled scores; may be NULL */
    int64_t     T_span;       /* = win_off[w_end] - win_off[w_begin] */
    const int32_t* d_win_off; /* device [M+1] from focus_layout */
    const int32_t* d_ring_off;/* device [M+1] from focus_layout */
    int32_t     n_windows;    /* M (the offsets arrays hold M+1 entries) */
    int32_t     w_begin, w_end;   /* 0 <= w_begin < w_end <= M */
    int32_t     max_rows;     /* >= every window's augmented row count in the span */
    float       scale;        /* softmax scale > 0, usually 1/sqrt(d) */
    uint32_t    flags;        /* FOCUS_PREFILL_* */
    void*       workspace;    /* device scratch, 16-byte aligned, or NULL (see focus_prefill_workspace_size) */
    size_t      workspace_bytes;  /* its size in bytes */
    const int32_t* h_k_per_window; /* optional HOST copy of cache->k_per_window (entries w_begin .. w_end-1
                                      read), or NULL; lets FOCUS_PREFILL_KMER_LOCAL use its k-mer-tiled
                                      kernel (below). Must hold the same values as the device schedule: a
                                      kernel that finds them different reports FOCUS_ERR_INVALID_ARG */
} focus_prefill_args;

/* Device workspace that lets focus_attn_prefill use its fastest kernels for these
 * arguments; 0 when none helps. Host only, no CUDA call; 0 also for arguments that
 * focus_attn_prefill would reject. Today only the rotary embedding
 * (cache->rope_theta > 0), outside the k-mer-tiled kernel's case (which rotates
 * in place), asks for one: 256 bytes of per-head counters (B x H int32, rounded up
 * to 256 bytes) followed by a rotated copy of the span's q rows ([B][H q_per_kv]
 * [T_span][d] bf16) and k rows ([B][H][T_span][d]).
 * With it, the q and k rows are each rotated once: by a pass of their own before
 * the attention (HBM-bound; the attention then runs as without the embedding, on
 * any kernel), or, for grouped-query heads (q_per_kv >= 2) on short work items
 * (the persistent kernel's case), by otherwise idle warps of the persistent
 * kernel itself, a head ahead of their use. Without it (NULL, or fewer bytes) the
 * call still succeeds and every CTA of the one-CTA-per-item kernel rotates the
 * tiles it loads. The contents need no initialisation and are scratch afterwards;
 * the caller owns the memory. */
size_t focus_prefill_workspace_size(const focus_cache* cache, const focus_prefill_args* args);

/* Use the legacy mma.sync kernel instead of the tcgen05/TMEM kernel (kept as the
 * comparison baseline; same results within rounding). It has no rotary
 * embedding: with cache->rope_theta > 0 the call returns FOCUS_ERR_UNSUPPORTED. */
#define FOCUS_PREFILL_LEGACY_MMA 1u

/* Main-text k-mer-local visibility (Sec. 3.2 "Visibility and summarization rule")
 * instead of the appendix mask. Row a of window w, in k-mer c = a / (k_w + 1)
 * (the whole window is one k-mer when k_w = 0), sees
 *   - window rows [c (k_w + 1), a]: the earlier rows of its own k-mer and itself,
 *   - the FOCUS rows of k-mers 0..c-1 of window w, read from the ring at rows
 *     [ring_off[w], ring_off[w] + c),
 *   - the carried boundary, ring row ring_off[w] - 1, when window w-1 has FOCUS
 *     rows (its last FOCUS row, S_{m,1} = S_{m-1,W}),
 * and nothing else. Requires cache->k_per_window (device [n_windows], the
 * layout's k schedule, n_windows >= w_end), cache->tail == 0 and a layout built
 * with tail 0 (FOCUS_ERR_UNSUPPORTED otherwise), and the FOCUS rows of windows
 * w_begin-1 .. w_end-1 already in the ring: compact before this call, also when
 * streaming. Not combinable with FOCUS_PREFILL_LEGACY_MMA (FOCUS_ERR_UNSUPPORTED). */
#define FOCUS_PREFILL_KMER_LOCAL 2u

/* Row a of window w (a = in-window augmented offset) gets
 *   o = softmax_j(scale * q·k_j) v_j over j ∈ ring[0, ring_off[w]) ∪ window rows [0, a]
 * and lse = ln Σ_j exp(scale * q·k_j). The ring rows are cache->ring_k/ring_v of the
 * same (b, h); ring_off[w] <= C_ring is required for every window of the span.
 * Masked-parallel use: bulk-compact all summaries first, then one call over all
 * windows. Streaming use: one call per window, then compact that window.
 * Keys are read in 128-row tiles and masked keys get weight 0, so every row of
 * ring_k/ring_v [0, C_ring) and of k/v [0, T_span) must hold finite values (a
 * zero-initialised cache does). Unknown flag bits: FOCUS_ERR_INVALID_ARG. */
focus_status focus_attn_prefill(const focus_cache* cache, const focus_prefill_args* args,
                                cudaStream_t stream);

/* Which kernel focus_attn_prefill launches for these arguments. Host only: no
 * device work, no CUDA call; the arguments are checked as focus_attn_prefill
 * checks them (same return codes). *kernel receives
 *   FOCUS_PREFILL_KERNEL_LEGACY      the mma.sync kernel (FOCUS_PREFILL_LEGACY_MMA),
 *   FOCUS_PREFILL_KERNEL_PERSISTENT  the tcgen05 kernel with one CTA per SM walking
 *                                    the work items (two 128-row Q tiles of a window
 *                                    each): appendix mask and
 *                                    cache->C_ring + args->max_rows <= 4096 (short
 *                                    items, whose start-up and epilogue it overlaps),
 *   FOCUS_PREFILL_KERNEL_PER_ITEM    the tcgen05 kernel with one CTA per work item
 *                                    (every other case).
 *   FOCUS_PREFILL_KERNEL_KMER        the FOCUS_PREFILL_KMER_LOCAL mode with query tiles cut at
 *                                    k-mer boundaries (one CTA per SM walking them): each tile's
 *                                    keys, its k-mers' rows plus the few ring rows they see, fit one
 *                                    128-row K/V tile. Taken when args->h_k_per_window is given and
 *                                    over the span's windows every k-mer
 *                                    has at most 128 - RB rows, where RB (a multiple of 8, <= 64)
 *                                    bounds the ring rows a tile sees: the boundary plus one FOCUS
 *                                    row per k bases, 1 + ceil(max_rows / k_w); and the launch has at
 *                                    least 2,048 work items (tiles x query heads x sequences).
 * With the rotary embedding the k-mer-tiled kernel rotates its tiles in place
 * (no workspace). Otherwise, with focus_prefill_workspace_size(cache, args) bytes
 * of workspace, the kernel is the one the same arguments take without the
 * embedding, and FOCUS_PREFILL_KERNEL_ROTATION_PASS is or-ed into *kernel when a
 * rotation pass runs before it (every case but grouped-query heads on the
 * persistent kernel, which rotates q and k itself); without the workspace the
 * rotary embedding takes the one-CTA-per-item kernel.
 * The tcgen05 kernels compute the same rows (within rounding order). */
#define FOCUS_PREFILL_KERNEL_LEGACY 0
#define FOCUS_PREFILL_KERNEL_PER_ITEM 1
#define FOCUS_PREFILL_KERNEL_PERSISTENT 2
#define FOCUS_PREFILL_KERNEL_KMER 3
#define FOCUS_PREFILL_KERNEL_ROTATION_PASS 16
focus_status focus_prefill_kernel(const focus_cache* cache, const focus_prefill_args* args, int32_t* kernel);

/* ------------------------------------------------------------------------ */
/* focus_prefill_host — the masked-parallel prefill (App. A.1) of a layer    */
/* whose inputs and outputs are in host memory.                             */
/* ------------------------------------------------------------------------ */
typedef struct focus_prefill_host_args {
    /* host memory; pinned (cudaHostAlloc / cudaHostRegister) for the copies to
     * overlap the kernels. Shapes as for focus_layout and focus_attn_prefill over
     * all windows (T = layout->T, g = cache->q_per_kv, at least 1): */
    const uint8_t* h_nt;      /* [B][n_nt] nucleotide ids */
    const void*    h_q;       /* bf16 [B][H g][T][d] */
    const void*    h_k;       /* bf16 [B][H][T][d] */
    const void*    h_v;       /* bf16 [B][H][T][d] */
    void*          h_o;       /* bf16 [B][H g][T][d], written */
    float*         h_lse;     /* fp32 [B][H g][T], written; may be NULL (then d_lse may be too) */
    /* device buffers of the same shapes, caller-owned (reused across calls) */
    uint8_t* d_nt;
    void*    d_q;
    void*    d_k;
    void*    d_v;
    void*    d_o;
    float*   d_lse;
    /* the layout, as for focus_layout / focus_layout_sched (d_W_sched NULL: windows
     * of W bases); layout->tok is written from d_nt (B rows) */
    int64_t  n_nt;
    int32_t  W;
    const int32_t* d_W_sched;
    int32_t  n_windows;
    const int32_t* d_k_sched;
    uint32_t layout_flags;
    int32_t  tail;
    const focus_layout_out* layout;
    int32_t  max_rows;        /* from focus_layout_size */
    float    scale;           /* softmax scale > 0 */
    uint32_t prefill_flags;   /* FOCUS_PREFILL_* */
    void*    workspace;       /* as in focus_prefill_args, shared by the parts in turn (its size for the
                                 whole cache covers every part), or NULL */
    size_t   workspace_bytes;
    int32_t  groups;          /* parts the heads (B = 1) or the sequences (B > 1) are cut into, >= 1 */
    cudaStream_t copy_in;     /* two streams of the caller, other than `stream`, for the copies in and out */
    cudaStream_t copy_out;
} focus_prefill_host_args;

/* The same computation as focus_layout + focus_kv_compact (bulk, all windows) +
 * focus_attn_prefill (all windows), from and to host memory: the token ids are
 * copied in and the layout built once; then for each of `groups` parts (K/V heads
 * [h0, h1) of the one sequence when B = 1, else sequences [b0, b1)) the part's q,
 * k, v are copied in on copy_in, its compaction and attention run on `stream`,
 * and its o and lse are copied out on copy_out, so that one part's copies overlap
 * the other parts' kernels and copies. One cudaMemcpyAsync per tensor and part
 * (a part is contiguous in every tensor). Outputs equal those of the device-buffer
 * calls bit for bit. Asynchronous: once `stream` has reached the end of the call,
 * so have the copies out (the call makes `stream` wait for copy_out); the device
 * buffers may be reused from there. The call creates and releases its own CUDA
 * events (no device memory). Argument errors as for the three calls it makes,
 * plus FOCUS_ERR_INVALID_ARG for missing pointers, groups < 1, or copy streams
 * equal to `stream`. Passage: App. A.1 "Cross-window consistency" (the
 * masked-parallel form) and App. A, "KV compression and budget". */
focus_status focus_prefill_host(const focus_cache* cache, const focus_prefill_host_args* args, cudaStream_t stream);

/* ------------------------------------------------------------------------ */
/* focus_attn_decode — one new token per sequence against the compressed    */
/* cache (App. A.2; decoding keeps the base decoder's interface).           */
/* ------------------------------------------------------------------------ */

/* Bytes of device workspace focus_attn_decode needs for this cache shape. */
size_t focus_decode_workspace_size(const focus_cache* cache);

/* For each (b, h): append k_new/v_new at window row win_fill[b], then
 *   o = softmax over ring[0, ring_len[b]) ∪ window[0, win_fill[b]] (itself included),
 * and increment win_fill[b]. q/k_new/v_new/o: device bf16 [B][H][d]; lse: device fp32
 * [B][H] or NULL. workspace: device, >= focus_decode_workspace_size(cache) bytes,
 * 16-byte aligned; its contents need no initialisation and are scratch afterwards.
 * If the window buffer of sequence b is already full (win_fill[b] == that window's
 * augmented size, or == C_win) the sequence is skipped and the status word is set to
 * FOCUS_ERR_CAPACITY: call focus_kv_compact between steps. */
focus_status focus_attn_decode(const focus_cache* cache, const void* q, const void* k_new,
                               const void* v_new, float scale, void* o, float* lse,
                               void* workspace, size_t workspace_bytes, cudaStream_t stream);

/* Allocation-free variant of focus_attn_decode. The paper has no counterpart:
 * this entry point exists for callers that cannot hand the library scratch
 * memory, e.g. a plugin inside a host runtime that owns all device memory and
 * passes in only its input and output buffers, or a serving loop that must not
 * call cudaMalloc/cudaFree (which can synchronise the device) between steps.
 *
 * Computes exactly what focus_attn_decode computes, with the same arguments
 * minus the workspace. The split-K partials go to a fixed array of
 * FOCUS_DECODE_NOALLOC_SCRATCH_BYTES inside the library, which every GPU that
 * loads the library holds until the process exits. The call allocates nothing.
 *   - If the cache needs more scratch than that (focus_decode_workspace_size(cache)
 *     > FOCUS_DECODE_NOALLOC_SCRATCH_BYTES; batch 64 x 32 heads at d = 128 with
 *     about 12k ring + window rows needs 12.8 MB) it returns FOCUS_ERR_CAPACITY
 *     and launches nothing: use focus_attn_decode with a workspace instead.
 *   - All calls on a device share the one array. Calls whose kernels overlap on
 *     the GPU (different streams without ordering between them) race on it and
 *     give wrong results; calls ordered on one stream are safe. The array keeps
 *     the previous call's contents; this needs no clearing, because every split
 *     writes its partial before the merge reads it.
 *   - The first call on each device looks up the array's device address (with
 *     that device current) and keeps it; make that first call before capturing
 *     any stream. */
#define FOCUS_DECODE_NOALLOC_SCRATCH_BYTES (16u << 20)

focus_status focus_attn_decode_noalloc(const focus_cache* cache, const void* q, const void* k_new,
                                       const void* v_new, float scale, void* o, float* lse,
                                       cudaStream_t stream);

/* ------------------------------------------------------------------------ */
/* focus_kv_compact — KV retention after a window (App. A, "KV compression  */
/* and budget"; Sec. 3.2 "KV retention and memory profile").               */
/* ------------------------------------------------------------------------ */
typedef struct focus_compact_args {
    /* Bulk mode (src_k != NULL): gather the FOCUS rows of windows [w_begin, w_end)
     * from an augmented K/V tensor into ring rows [ring_off[w_begin], ring_off[w_end])
     * of every (b, h), then set ring_len[b] = ring_off[w_end] for all b. */
    const void* src_k;        /* device bf16 [B][H][src_T][d]; NULL selects window mode */
    const void* src_v;        /* device bf16 [B][H][src_T][d] */
    int64_t     src_T;        /* rows per (b, h) in src */
    int64_t     src_row0;     /* augmented index of src row 0 (e.g. win_off[w_begin]) */
    const int32_t* d_sum_idx; /* device [R] from focus_layout */
    const int32_t* d_ring_off;/* device [M+1] from focus_layout */
    int32_t     n_windows;    /* M (the offsets arrays hold M+1 entries) */
    int32_t     w_begin, w_end;   /* 0 <= w_begin <= w_end <= M */
    /* Window mode (src_k == NULL): for each sequence b whose window buffer is full
     * (win_fill[b] == W + ceil(W / k_{win_idx[b]})), append that window's kept rows
     * (its FOCUS rows and its last cache->tail bases, in augmented order) to the ring
     * at ring_len[b], advance ring_len[b], reset win_fill[b] to 0 and increment
     * win_idx[b]. Sequences with a partly filled window are untouched. */
} focus_compact_args;

focus_status focus_kv_compact(const focus_cache* cache, const focus_compact_args* args,
                              cudaStream_t stream);

/* Self-test of the failure path (no fault, no hang): one CTA waits, with the
 * bounded mbarrier wait every kernel of this library uses, on a barrier nothing
 * arrives on; after limit_ns it gives up and sets the device status word to
 * FOCUS_ERR_TIMEOUT, as a kernel whose copies or MMAs never completed would. The
 * context stays usable. Kernels that find FOCUS_ERR_TIMEOUT already set skip their
 * work (so that a systematic stall costs one round of waits), so clear the word
 * (focus_get_device_status with clear != 0) before further calls.
 * 0 < limit_ns <= 10 s, else FOCUS_ERR_INVALID_ARG. Asynchronous on `stream`. */
focus_status focus_selftest_timeout(uint64_t limit_ns, cudaStream_t stream);

/* ------------------------------------------------------------------------ */
/* focus_embed_tokens — input rows of the augmented sequence (Sec. 3.2      */
/* "Setup and tokens": the FOCUS summary is a learned token inserted after  */
/* every k-mer; App. A: the inserted tokens take positions of their own).   */
/* ------------------------------------------------------------------------ */
/* out[i][:] = table[tok[i]][:] for i < n_rows: the token stream focus_layout
 * writes (nucleotide ids 0..3, FOCUS_SUMMARY_TOKEN for a summary) looked up in an
 * embedding table whose row FOCUS_SUMMARY_TOKEN is the summary token's vector.
 * Device pointers, caller-owned: d_tok uint8 [n_rows] (e.g. layout tok, B x T
 * rows), d_table bf16 [n_tokens][D], d_out bf16 [n_rows][D]; D a positive
 * multiple of 8 and both bf16 pointers 16-byte aligned (else
 * FOCUS_ERR_UNSUPPORTED), 1 <= n_tokens <= 256. A token >= n_tokens writes a zero
 * row and sets the device status word to FOCUS_ERR_INVALID_ARG. n_rows = 0 is a
 * no-op. Asynchronous on `stream`. */
focus_status focus_embed_tokens(const uint8_t* d_tok, int64_t n_rows, const void* d_table, int32_t n_tokens,
                                int32_t D, void* d_out, cudaStream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* FOCUS_H_ */
