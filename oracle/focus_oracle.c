/*
 * FOCUS oracle: plain, slow, fp64 CPU statement of what the compressed-context
 * attention path computes (arXiv 2511.14694, Appendix A).
 *
 * TEST INFRASTRUCTURE ONLY. The test suite, the smoke check and the benchmark's
 * CPU-baseline leg are the only users. The CUDA library never includes, links
 * or calls this file, and this file shares nothing with it.
 *
 * Conventions
 *   - Nucleotide ids are 0..3 (A, C, G, T); the reserved summary-token id is 4
 *     (Table "Full configuration" lists a reserved id for the FOCUS token).
 *   - Indices are 0-based. Window w covers bases [w*W, min((w+1)*W, N)), the
 *     0-based form of I_w = [(w-1)W+1, wW] ∩ [1, L]  (App. A, first display).
 *   - Q/K/V arrive as raw bf16 bit patterns (uint16) exactly as the GPU sees
 *     them; each is widened to fp64 here (bf16 -> fp32 is exact, fp32 -> fp64
 *     is exact). All arithmetic after that is fp64.
 *   - Softmax scale is a caller argument; LSE is the natural log of the sum of
 *     exponentials of the scaled scores.
 *
 * KV retention keeps each window's FOCUS rows and, optionally, a boundary
 * tail: the last `tail` ordinary (base) rows of the window (App. A allows a
 * short boundary tail besides the FOCUS rows; App. A.2). tail = 0 is the paper's default.
 * A kept row is visible to every later window.
 *
 * Every loop below runs in the order the paper states the operation; nothing is
 * blocked, fused or reordered.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define FO_SUMMARY_TOKEN 4

static double bf16_to_f64(uint16_t bits) {
    uint32_t u = ((uint32_t)bits) << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* ------------------------------------------------------------------------- */
/* Token layout (App. A: windows I_w, M = ceil(L/W), B_w = ceil(|I_w|/k),     */
/* one FOCUS token per k real bases at the right boundary of its k-mer,       */
/* each FOCUS token taking a position of its own, as a base does).           */
/* ------------------------------------------------------------------------- */

/* Does a summary follow the base at in-window offset o (0-based) of a window
 * holding n bases with cadence k? A summary closes every full k-mer, and the
 * partial k-mer at the window's end when `close_partial` is set (the ceil in
 * B_w = ceil(|I_w|/k)). k == 0 means "no summaries" (compression disabled). */
static int summary_after(int64_t o, int64_t n, int32_t k, int close_partial) {
    if (k <= 0) return 0;
    if ((o + 1) % k == 0) return 1;
    return (o == n - 1) && close_partial;
}

/* Is the base at in-window offset o of an n-base window in its boundary tail? */
static int in_tail(int64_t o, int64_t n, int32_t tail) { return tail > 0 && o >= n - tail; }

/* Window w covers the W_sched[w] bases after the previous windows' (the last
 * one may hold fewer): windows of one length W are W_sched[w] = W, and adaptive
 * windowing (choosing W, like k, per region; Sec. 5) gives each its own.
 * Returns 0 if the schedule of M windows covers exactly N bases with every
 * window non-empty, else -1. */
static int32_t check_windows(int64_t N, int32_t M, const int32_t* W_sched) {
    if (N < 0 || M < 0 || (M > 0 && !W_sched)) return -1;
    int64_t start = 0;
    for (int32_t w = 0; w < M; ++w) {
        if (W_sched[w] <= 0 || start >= N) return -1;
        start += W_sched[w];
    }
    return start >= N ? 0 : -1;
}

static int64_t window_bases(int64_t N, int64_t start, int32_t W) { return (N - start < W) ? (N - start) : W; }

/* Sizes of the augmented layout. Returns T (augmented length) and writes R
 * (rows retained after the last window: summaries plus boundary tails).
 * Returns -1 on bad arguments. */
int64_t fo_layout_size_sched(int64_t N, int32_t M, const int32_t* W_sched, const int32_t* k_sched,
                             int32_t close_tail, int32_t tail, int64_t* R_out) {
    if (tail < 0 || check_windows(N, M, W_sched) != 0) return -1;
    int64_t T = 0, R = 0, start = 0;
    for (int32_t w = 0; w < M; ++w) {
        int64_t n = window_bases(N, start, W_sched[w]);
        int close = (w < M - 1) || close_tail;
        for (int64_t o = 0; o < n; ++o) {
            T += 1;
            if (in_tail(o, n, tail)) R += 1;
            if (summary_after(o, n, k_sched[w], close)) { T += 1; R += 1; }
        }
        start += W_sched[w];
    }
    if (R_out) *R_out = R;
    return T;
}

/* Full layout walk. For every augmented index t:
 *   kind[t]  0 = ordinary base, 1 = FOCUS summary
 *   src[t]   nucleotide index of the base (for a summary: its k-mer's last base)
 *   pos[t]   position id = t (a summary has a position of its own)
 *   win[t]   window id w
 *   tok[b*T + t]  nucleotide id nt[b*N + src] for bases, 4 for summaries
 *                 (written only when nt and tok are both non-NULL)
 *   keep[t]  1 if KV retention keeps the row (a summary, or a boundary-tail base)
 * plus win_off[M+1] (first augmented index of each window, win_off[M] = T),
 * ring_off[M+1] (rows retained before each window, ring_off[M] = R),
 * sum_idx[R] (augmented index of each retained row, in order) and, if not NULL,
 * base_off[M+1] (first base of each window, base_off[M] = N).
 * Returns T, or -1 on bad arguments. */
int64_t fo_layout_sched(int64_t N, int32_t M, const int32_t* W_sched, const int32_t* k_sched,
                        int32_t close_tail, int32_t tail, int32_t B, const uint8_t* nt,
                        uint8_t* kind, int32_t* src, int32_t* pos, int32_t* win,
                        uint8_t* tok, uint8_t* keep, int32_t* win_off, int32_t* ring_off,
                        int32_t* sum_idx, int32_t* base_off) {
    int64_t R_total = 0;
    int64_t T_total = fo_layout_size_sched(N, M, W_sched, k_sched, close_tail, tail, &R_total);
    if (T_total < 0) return -1;
    int64_t t = 0, r = 0, start = 0;
    for (int32_t w = 0; w < M; ++w) {
        int64_t n = window_bases(N, start, W_sched[w]);
        int close = (w < M - 1) || close_tail;
        win_off[w] = (int32_t)t;
        ring_off[w] = (int32_t)r;
        if (base_off) base_off[w] = (int32_t)start;
        for (int64_t o = 0; o < n; ++o) {
            int64_t base = start + o;
            kind[t] = 0; src[t] = (int32_t)base; pos[t] = (int32_t)t; win[t] = w;
            keep[t] = (uint8_t)in_tail(o, n, tail);
            if (keep[t]) { sum_idx[r] = (int32_t)t; r += 1; }
            if (nt && tok)
                for (int32_t b = 0; b < B; ++b) tok[(int64_t)b * T_total + t] = nt[(int64_t)b * N + base];
            t += 1;
            if (summary_after(o, n, k_sched[w], close)) {
                kind[t] = 1; src[t] = (int32_t)base; pos[t] = (int32_t)t; win[t] = w;
                keep[t] = 1;
                if (nt && tok)
                    for (int32_t b = 0; b < B; ++b) tok[(int64_t)b * T_total + t] = FO_SUMMARY_TOKEN;
                sum_idx[r] = (int32_t)t;
                r += 1;
                t += 1;
            }
        }
        start += W_sched[w];
    }
    win_off[M] = (int32_t)t;
    ring_off[M] = (int32_t)r;
    if (base_off) base_off[M] = (int32_t)N;
    return t;
}

/* Windows of one length W: M = ceil(N/W) windows of W bases (App. A, I_w). */
static int32_t* fixed_windows(int64_t N, int32_t W, int32_t M) {
    if (W <= 0 || M < 0 || (int64_t)M != (N + W - 1) / W) return NULL;
    int32_t* s = (int32_t*)malloc(sizeof(int32_t) * (size_t)(M > 0 ? M : 1));
    for (int32_t w = 0; w < M; ++w) s[w] = W;
    return s;
}

int64_t fo_layout_size(int64_t N, int32_t W, int32_t M, const int32_t* k_sched,
                       int32_t close_tail, int32_t tail, int64_t* R_out) {
    int32_t* Ws = fixed_windows(N, W, M);
    if (!Ws) return -1;
    int64_t T = fo_layout_size_sched(N, M, Ws, k_sched, close_tail, tail, R_out);
    free(Ws);
    return T;
}

int64_t fo_layout(int64_t N, int32_t W, int32_t M, const int32_t* k_sched,
                  int32_t close_tail, int32_t tail, int32_t B, const uint8_t* nt,
                  uint8_t* kind, int32_t* src, int32_t* pos, int32_t* win,
                  uint8_t* tok, uint8_t* keep, int32_t* win_off, int32_t* ring_off,
                  int32_t* sum_idx) {
    int32_t* Ws = fixed_windows(N, W, M);
    if (!Ws) return -1;
    int64_t T = fo_layout_sched(N, M, Ws, k_sched, close_tail, tail, B, nt, kind, src, pos, win, tok, keep,
                                win_off, ring_off, sum_idx, NULL);
    free(Ws);
    return T;
}

/* ------------------------------------------------------------------------- */
/* Softmax attention of one query row over an explicit, ordered list of key   */
/* rows: s_j = scale * <q, k_j>, m = max s, l = sum exp(s_j - m),             */
/* o = sum exp(s_j - m) v_j / l, LSE = m + ln l.                              */
/* ------------------------------------------------------------------------- */

/* The part after the dot products: s[j] holds <q, k_j> on entry. */
static void softmax_of_dots(int32_t d, int64_t n_keys, double* s, const uint16_t* const* vrows,
                            double scale, double* o, double* lse) {
    double m = -INFINITY;
    for (int64_t j = 0; j < n_keys; ++j) {
        s[j] = scale * s[j];
        if (s[j] > m) m = s[j];
    }
    double l = 0.0;
    for (int32_t c = 0; c < d; ++c) o[c] = 0.0;
    for (int64_t j = 0; j < n_keys; ++j) {
        double p = exp(s[j] - m);
        l += p;
        for (int32_t c = 0; c < d; ++c) o[c] += p * bf16_to_f64(vrows[j][c]);
    }
    for (int32_t c = 0; c < d; ++c) o[c] /= l;
    *lse = m + log(l);
}

static void softmax_row(int32_t d, const uint16_t* q, int64_t n_keys,
                        const uint16_t* const* krows, const uint16_t* const* vrows,
                        double scale, double* o, double* lse) {
    double* qd = (double*)malloc(sizeof(double) * (size_t)d);
    double* s = (double*)malloc(sizeof(double) * (size_t)(n_keys > 0 ? n_keys : 1));
    for (int32_t c = 0; c < d; ++c) qd[c] = bf16_to_f64(q[c]);
    for (int64_t j = 0; j < n_keys; ++j) {
        double dot = 0.0;
        for (int32_t c = 0; c < d; ++c) dot += qd[c] * bf16_to_f64(krows[j][c]);
        s[j] = dot;
    }
    softmax_of_dots(d, n_keys, s, vrows, scale, o, lse);
    free(s);
    free(qd);
}

/* ------------------------------------------------------------------------- */
/* Masked-parallel form (App. A.1, "Cross-window consistency" (ii), with the  */
/* visible set of Eq. focus-attn / C(t)): row i sees key j iff j <= i and     */
/* (j is in the same window as i, or j is a retained row: a FOCUS token or a  */
/* boundary-tail base; keep[] marks them).                                     */
/*                                                                            */
/* q, k, v: [n_heads][T][d] bf16 bits. Computes the requested rows only:     */
/* row r is (head row_head[r], augmented index row_idx[r]). Outputs o[r][d],  */
/* lse[r].                                                                    */
/* ------------------------------------------------------------------------- */
void fo_attn_rows(int64_t T, int32_t d, const uint8_t* keep, const int32_t* win,
                  const uint16_t* q, const uint16_t* k, const uint16_t* v,
                  double scale, int64_t n_rows, const int64_t* row_head,
                  const int64_t* row_idx, double* o, double* lse) {
#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t r = 0; r < n_rows; ++r) {
        int64_t h = row_head[r], i = row_idx[r];
        const uint16_t* kh = k + (size_t)h * (size_t)T * (size_t)d;
        const uint16_t* vh = v + (size_t)h * (size_t)T * (size_t)d;
        const uint16_t** kr = (const uint16_t**)malloc(sizeof(void*) * (size_t)(i + 1));
        const uint16_t** vr = (const uint16_t**)malloc(sizeof(void*) * (size_t)(i + 1));
        int64_t n = 0;
        for (int64_t j = 0; j <= i; ++j) {
            int visible = (win[j] == win[i]) || (keep[j] == 1);
            if (!visible) continue;
            kr[n] = kh + (size_t)j * d;
            vr[n] = vh + (size_t)j * d;
            n += 1;
        }
        softmax_row(d, q + ((size_t)h * (size_t)T + (size_t)i) * d, n, kr, vr, scale,
                    o + (size_t)r * d, lse + r);
        free(kr);
        free(vr);
    }
}

/* ------------------------------------------------------------------------- */
/* Sequential form (App. A.1 (i); App. A.2 "Streaming with controlled         */
/* memory"): windows in order; each row of window w attends to the retained   */
/* FOCUS KV of earlier windows and to the rows of window w up to itself;      */
/* after window w its ordinary KV is dropped and its FOCUS KV is appended to   */
/* the retained set (App. A, "KV compression and budget").                    */
/*                                                                            */
/* One head: q, k, v are [T][d] bf16 bits; win_off[M+1] gives window rows;    */
/* keep[T] marks retained rows. want[M] (NULL = all) selects the windows whose */
/* outputs are computed; retention runs for every window regardless. Writes   */
/* o[T][d], lse[T] for computed windows (others untouched) and the retained   */
/* KV (ring_k/ring_v, [ring_cap][d]) with its length in *R_out.               */
/* Returns 0, or -1 if ring_cap is too small.                                 */
/* ------------------------------------------------------------------------- */
int32_t fo_prefill_sequential(int32_t d, int32_t M, const int32_t* win_off,
                              const uint8_t* keep, const uint16_t* q,
                              const uint16_t* k, const uint16_t* v, double scale,
                              const uint8_t* want, double* o, double* lse,
                              uint16_t* ring_k, uint16_t* ring_v, int64_t ring_cap,
                              int64_t* R_out) {
    int64_t R = 0;
    for (int32_t w = 0; w < M; ++w) {
        int64_t a = win_off[w], e = win_off[w + 1];
        if (!want || want[w]) {
#pragma omp parallel for schedule(dynamic, 8)
            for (int64_t i = a; i < e; ++i) {
                int64_t nk = R + (i - a + 1);
                const uint16_t** kr = (const uint16_t**)malloc(sizeof(void*) * (size_t)nk);
                const uint16_t** vr = (const uint16_t**)malloc(sizeof(void*) * (size_t)nk);
                int64_t n = 0;
                for (int64_t j = 0; j < R; ++j) {          /* retained history */
                    kr[n] = ring_k + (size_t)j * d;
                    vr[n] = ring_v + (size_t)j * d;
                    n += 1;
                }
                for (int64_t j = a; j <= i; ++j) {          /* current window, causal */
                    kr[n] = k + (size_t)j * d;
                    vr[n] = v + (size_t)j * d;
                    n += 1;
                }
                softmax_row(d, q + (size_t)i * d, n, kr, vr, scale, o + (size_t)i * d, lse + i);
                free(kr);
                free(vr);
            }
        }
        /* window finished: keep FOCUS KV (and the boundary tail), drop the rest */
        for (int64_t j = a; j < e; ++j) {
            if (keep[j] != 1) continue;
            if (R >= ring_cap) return -1;
            memcpy(ring_k + (size_t)R * d, k + (size_t)j * d, sizeof(uint16_t) * (size_t)d);
            memcpy(ring_v + (size_t)R * d, v + (size_t)j * d, sizeof(uint16_t) * (size_t)d);
            R += 1;
        }
    }
    *R_out = R;
    return 0;
}

/* ------------------------------------------------------------------------- */
/* Decode (App. A.2): one new token per sequence. Its K/V are appended to the */
/* current window; its query attends to the retained FOCUS KV (ring, R rows)  */
/* and to the current window's rows up to and including itself.              */
/*                                                                            */
/* Batched over n independent (sequence, head) streams: stream s has          */
/* ring_k/ring_v rows [s*ring_stride, +R[s]) and window rows                   */
/* [s*win_stride, +fill[s]) (fill BEFORE the append). q/k_new/v_new: [n][d].  */
/* The append itself is the caller's (this routine reads k_new/v_new as the   */
/* last visible row). Outputs o[n][d], lse[n].                                */
/* ------------------------------------------------------------------------- */
void fo_decode(int32_t d, int64_t n, const uint16_t* ring_k, const uint16_t* ring_v,
               int64_t ring_stride, const int64_t* R, const uint16_t* win_k,
               const uint16_t* win_v, int64_t win_stride, const int64_t* fill,
               const uint16_t* q, const uint16_t* k_new, const uint16_t* v_new,
               double scale, double* o, double* lse) {
#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t s = 0; s < n; ++s) {
        int64_t nk = R[s] + fill[s] + 1;
        const uint16_t** kr = (const uint16_t**)malloc(sizeof(void*) * (size_t)nk);
        const uint16_t** vr = (const uint16_t**)malloc(sizeof(void*) * (size_t)nk);
        int64_t c = 0;
        for (int64_t j = 0; j < R[s]; ++j) {
            kr[c] = ring_k + ((size_t)s * ring_stride + (size_t)j) * d;
            vr[c] = ring_v + ((size_t)s * ring_stride + (size_t)j) * d;
            c += 1;
        }
        for (int64_t j = 0; j < fill[s]; ++j) {
            kr[c] = win_k + ((size_t)s * win_stride + (size_t)j) * d;
            vr[c] = win_v + ((size_t)s * win_stride + (size_t)j) * d;
            c += 1;
        }
        kr[c] = k_new + (size_t)s * d;
        vr[c] = v_new + (size_t)s * d;
        c += 1;
        softmax_row(d, q + (size_t)s * d, c, kr, vr, scale, o + (size_t)s * d, lse + s);
        free(kr);
        free(vr);
    }
}

/* In-window offsets (augmented, 0-based) of the rows KV retention keeps in one
 * window of n bases with cadence k: its FOCUS rows and its last `tail` bases
 * (App. A, "KV compression and budget"), in augmented order. Writes up to cap
 * offsets; returns their count. */
int32_t fo_window_retained_rows(int64_t n, int32_t k, int32_t close_partial, int32_t tail,
                                int32_t* out, int32_t cap) {
    int64_t t = 0;
    int32_t c = 0;
    for (int64_t o = 0; o < n; ++o) {
        if (in_tail(o, n, tail)) {
            if (c < cap) out[c] = (int32_t)t;
            c += 1;
        }
        t += 1;
        if (summary_after(o, n, k, close_partial)) {
            if (c < cap) out[c] = (int32_t)t;
            c += 1;
            t += 1;
        }
    }
    return c;
}

/* ------------------------------------------------------------------------- */
/* k-mer membership (Sec. 3.2 "Setup and tokens": a base belongs to exactly   */
/* one k-mer; the FOCUS token S_i closes the k-mer B_i to its left). kmer[t] */
/* is the 0-based index, within its window, of the k-mer row t belongs to: a  */
/* base's own k-mer, or for a FOCUS token the k-mer it summarises. With k = 0 */
/* (no summaries) the whole window is one segment, index 0. Returns T or -1.  */
/* ------------------------------------------------------------------------- */
int64_t fo_layout_kmer_sched(int64_t N, int32_t M, const int32_t* W_sched, const int32_t* k_sched,
                             int32_t close_tail, int32_t* kmer) {
    if (fo_layout_size_sched(N, M, W_sched, k_sched, close_tail, 0, NULL) < 0) return -1;
    int64_t t = 0, start = 0;
    for (int32_t w = 0; w < M; ++w) {
        int64_t n = window_bases(N, start, W_sched[w]);
        int close = (w < M - 1) || close_tail;
        int32_t c = 0;
        for (int64_t o = 0; o < n; ++o) {
            kmer[t++] = c;
            if (summary_after(o, n, k_sched[w], close)) {
                kmer[t++] = c;
                c += 1;
            }
        }
        start += W_sched[w];
    }
    return t;
}

int64_t fo_layout_kmer(int64_t N, int32_t W, int32_t M, const int32_t* k_sched,
                       int32_t close_tail, int32_t* kmer) {
    int32_t* Ws = fixed_windows(N, W, M);
    if (!Ws) return -1;
    int64_t T = fo_layout_kmer_sched(N, M, Ws, k_sched, close_tail, kmer);
    free(Ws);
    return T;
}

/* ------------------------------------------------------------------------- */
/* Main-text visibility (Sec. 3.2 "Visibility and summarization rule"), the  */
/* k-mer-local mask. Row i of window w sees key j <= i iff                     */
/*   - j is in window w and in the same k-mer as i (a base sees the earlier   */
/*     bases of its own k-mer; a FOCUS token sees the k bases it summarises), */
/*   - or j is a FOCUS token of window w (the preceding in-window summaries), */
/*   - or j is the carried boundary of window w: the last FOCUS token of      */
/*     window w-1 (S_{m,1} == S_{m-1,W}, "Windowing with a shared boundary"). */
/* Nothing else of earlier windows is visible. kind/win/kmer: the layout's   */
/* per-row arrays. Same row selection and outputs as fo_attn_rows.            */
/* ------------------------------------------------------------------------- */
void fo_attn_rows_kmer_local(int64_t T, int32_t d, const uint8_t* kind, const int32_t* win,
                             const int32_t* kmer, const uint16_t* q, const uint16_t* k,
                             const uint16_t* v, double scale, int64_t n_rows,
                             const int64_t* row_head, const int64_t* row_idx, double* o,
                             double* lse) {
    int32_t M = T > 0 ? win[T - 1] + 1 : 0;
    int64_t* last_focus = (int64_t*)malloc(sizeof(int64_t) * (size_t)(M > 0 ? M : 1));
    for (int32_t w = 0; w < M; ++w) last_focus[w] = -1;
    for (int64_t j = 0; j < T; ++j)
        if (kind[j] == 1) last_focus[win[j]] = j;
#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t r = 0; r < n_rows; ++r) {
        int64_t h = row_head[r], i = row_idx[r];
        const uint16_t* kh = k + (size_t)h * (size_t)T * (size_t)d;
        const uint16_t* vh = v + (size_t)h * (size_t)T * (size_t)d;
        const uint16_t** kr = (const uint16_t**)malloc(sizeof(void*) * (size_t)(i + 1));
        const uint16_t** vr = (const uint16_t**)malloc(sizeof(void*) * (size_t)(i + 1));
        int64_t boundary = win[i] >= 1 ? last_focus[win[i] - 1] : -1;
        int64_t n = 0;
        for (int64_t j = 0; j <= i; ++j) {
            int same_window = win[j] == win[i];
            int visible = (same_window && kmer[j] == kmer[i]) || (same_window && kind[j] == 1) || j == boundary;
            if (!visible) continue;
            kr[n] = kh + (size_t)j * d;
            vr[n] = vh + (size_t)j * d;
            n += 1;
        }
        softmax_row(d, q + ((size_t)h * (size_t)T + (size_t)i) * d, n, kr, vr, scale,
                    o + (size_t)r * d, lse + r);
        free(kr);
        free(vr);
    }
    free(last_focus);
}

/* ------------------------------------------------------------------------- */
/* Rotary position embedding at the layout's position ids (RoFormer, Su et    */
/* al. 2021; the position id of a row is its augmented index: Sec. 3.2 gives  */
/* each FOCUS token a position of its own). Rotate-half pairing: for         */
/* i < d/2, the pair (x_i, x_{i+d/2}) is turned by the angle p * theta_i,     */
/* theta_i = base^(-2i/d):                                                    */
/*   y_i       = x_i cos(p theta_i) - x_{i+d/2} sin(p theta_i)                */
/*   y_{i+d/2} = x_{i+d/2} cos(p theta_i) + x_i sin(p theta_i)               */
/* x: [n][d] bf16 bits, pos[n]; y: [n][d] fp64.                               */
/* ------------------------------------------------------------------------- */
/* Round x to the nearest bf16 value (8 significant bits), ties to even, in one
 * step from fp64 (bf16 keeps fp32's exponent range; these values are normal). */
double fo_round_bf16(double x) {
    if (x == 0.0 || !isfinite(x)) return x;
    int e;
    double m = frexp(x, &e);                 /* x = m 2^e, 0.5 <= |m| < 1 */
    double r = nearbyint(ldexp(m, 8));       /* default rounding mode: to nearest, ties to even */
    return ldexp(r, e - 8);
}

/* round_bf16 != 0: each output is rounded once to bf16, the element type of the
 * rotated rows in a bf16 attention path. */
void fo_rope(int64_t n, int32_t d, const int64_t* pos, double base, int32_t round_bf16, const uint16_t* x,
             double* y) {
    int32_t h = d / 2;
    for (int64_t r = 0; r < n; ++r) {
        const uint16_t* xr = x + (size_t)r * d;
        double* yr = y + (size_t)r * d;
        for (int32_t i = 0; i < h; ++i) {
            double theta = pow(base, -2.0 * (double)i / (double)d);
            double a = (double)pos[r] * theta;
            double c = cos(a), s = sin(a);
            double lo = bf16_to_f64(xr[i]), hi = bf16_to_f64(xr[i + h]);
            yr[i] = lo * c - hi * s;
            yr[i + h] = hi * c + lo * s;
            if (round_bf16) {
                yr[i] = fo_round_bf16(yr[i]);
                yr[i + h] = fo_round_bf16(yr[i + h]);
            }
        }
    }
}

/* Softmax attention of one fp64 query over fp64 key rows (used where Q and K */
/* carry the rotary embedding).                                              */
static void softmax_row_f64(int32_t d, const double* q, int64_t n_keys, const double* const* krows,
                            const uint16_t* const* vrows, double scale, double* o, double* lse) {
    double* s = (double*)malloc(sizeof(double) * (size_t)(n_keys > 0 ? n_keys : 1));
    for (int64_t j = 0; j < n_keys; ++j) {
        double dot = 0.0;
        for (int32_t c = 0; c < d; ++c) dot += q[c] * krows[j][c];
        s[j] = dot;
    }
    softmax_of_dots(d, n_keys, s, vrows, scale, o, lse);
    free(s);
}

/* fo_attn_rows with fp64 queries and keys (e.g. after fo_rope): the same     */
/* visible set (App. A: same window, or a retained row), qf/kf [n_heads][T][d] */
/* fp64, v bf16 bits.                                                         */
void fo_attn_rows_f64(int64_t T, int32_t d, const uint8_t* keep, const int32_t* win, const double* qf,
                      const double* kf, const uint16_t* v, double scale, int64_t n_rows,
                      const int64_t* row_head, const int64_t* row_idx, double* o, double* lse) {
#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t r = 0; r < n_rows; ++r) {
        int64_t h = row_head[r], i = row_idx[r];
        const double* kh = kf + (size_t)h * (size_t)T * (size_t)d;
        const uint16_t* vh = v + (size_t)h * (size_t)T * (size_t)d;
        const double** kr = (const double**)malloc(sizeof(void*) * (size_t)(i + 1));
        const uint16_t** vr = (const uint16_t**)malloc(sizeof(void*) * (size_t)(i + 1));
        int64_t n = 0;
        for (int64_t j = 0; j <= i; ++j) {
            if (!((win[j] == win[i]) || (keep[j] == 1))) continue;
            kr[n] = kh + (size_t)j * d;
            vr[n] = vh + (size_t)j * d;
            n += 1;
        }
        softmax_row_f64(d, qf + ((size_t)h * (size_t)T + (size_t)i) * d, n, kr, vr, scale,
                        o + (size_t)r * d, lse + r);
        free(kr);
        free(vr);
    }
}

/* fo_decode with fp64 queries and keys: ring_k/win_k/k_new/q fp64 (already   */
/* rotated by the caller), values bf16 bits; otherwise identical.            */
void fo_decode_f64(int32_t d, int64_t n, const double* ring_k, const uint16_t* ring_v,
                   int64_t ring_stride, const int64_t* R, const double* win_k,
                   const uint16_t* win_v, int64_t win_stride, const int64_t* fill,
                   const double* q, const double* k_new, const uint16_t* v_new,
                   double scale, double* o, double* lse) {
#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t s = 0; s < n; ++s) {
        int64_t nk = R[s] + fill[s] + 1;
        const double** kr = (const double**)malloc(sizeof(void*) * (size_t)nk);
        const uint16_t** vr = (const uint16_t**)malloc(sizeof(void*) * (size_t)nk);
        int64_t c = 0;
        for (int64_t j = 0; j < R[s]; ++j) {
            kr[c] = ring_k + ((size_t)s * ring_stride + (size_t)j) * d;
            vr[c] = ring_v + ((size_t)s * ring_stride + (size_t)j) * d;
            c += 1;
        }
        for (int64_t j = 0; j < fill[s]; ++j) {
            kr[c] = win_k + ((size_t)s * win_stride + (size_t)j) * d;
            vr[c] = win_v + ((size_t)s * win_stride + (size_t)j) * d;
            c += 1;
        }
        kr[c] = k_new + (size_t)s * d;
        vr[c] = v_new + (size_t)s * d;
        c += 1;
        softmax_row_f64(d, q + (size_t)s * d, c, kr, vr, scale, o + (size_t)s * d, lse + s);
        free(kr);
        free(vr);
    }
}
