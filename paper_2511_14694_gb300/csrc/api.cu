// C ABI of libfocus.so (declared in include/focus.h): host-side argument
// checks, the per-device sticky status word, and dispatch to the kernels.
#include <math.h>
#include <mutex>

#include "common.cuh"

namespace {

// Sticky status word written by kernels (first error wins). One copy per device
// that loads the library; its device address is looked up once per device.
__device__ int32_t g_focus_status;

constexpr int kMaxDevices = 64;
int32_t* g_status_ptr[kMaxDevices];
std::mutex g_status_mu;

focus_status status_ptr(int32_t** out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return FOCUS_ERR_CUDA;
    std::lock_guard<std::mutex> lock(g_status_mu);
    if (!g_status_ptr[dev]) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_focus_status) != cudaSuccess) return FOCUS_ERR_CUDA;
        g_status_ptr[dev] = static_cast<int32_t*>(p);
    }
    *out = g_status_ptr[dev];
    return FOCUS_OK;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

focus_status from_cuda(cudaError_t e) { return e == cudaSuccess ? FOCUS_OK : FOCUS_ERR_CUDA; }

focus_status check_cache(const focus_cache* c, bool need_window) {
    if (!c) return FOCUS_ERR_INVALID_ARG;
    if (!isfinite(c->rope_theta) || c->rope_theta < 0.f) return FOCUS_ERR_INVALID_ARG;
    if (c->q_per_kv < 0 || c->q_per_kv > 64) return FOCUS_ERR_INVALID_ARG;
    if (c->B <= 0 || c->H <= 0 || c->C_ring < 0 || c->C_win < 0 || c->tail < 0) return FOCUS_ERR_INVALID_ARG;
    if (c->d != 64 && c->d != 128) return FOCUS_ERR_UNSUPPORTED;
    if ((int64_t)c->B > 65535 || (int64_t)c->H > 65535) return FOCUS_ERR_UNSUPPORTED;
    if (c->C_ring > 0 && (!c->ring_k || !c->ring_v)) return FOCUS_ERR_INVALID_ARG;
    if (c->ring_k && (!aligned16(c->ring_k) || !aligned16(c->ring_v))) return FOCUS_ERR_UNSUPPORTED;
    if (need_window) {
        if (!c->win_k || !c->win_v || !c->ring_len || !c->win_fill || !c->win_idx || !c->k_per_window)
            return FOCUS_ERR_INVALID_ARG;
        if ((c->W <= 0 && !c->W_per_window) || c->n_windows <= 0 || c->C_win <= 0) return FOCUS_ERR_INVALID_ARG;
        if (!aligned16(c->win_k) || !aligned16(c->win_v)) return FOCUS_ERR_UNSUPPORTED;
    }
    return FOCUS_OK;
}

}  // namespace

namespace focus {

void rope_table_fill(RopeTable* t, int d, float base) {
    const int h = d / 2;
    for (int i = 0; i < kRopeMaxPairs; ++i) t->theta[i] = i < h ? pow((double)base, -2.0 * i / d) : 0.0;
}

}  // namespace focus

extern "C" {

int32_t focus_version(void) { return 100; }

const char* focus_status_string(focus_status s) {
    switch (s) {
        case FOCUS_OK: return "ok";
        case FOCUS_ERR_INVALID_ARG: return "invalid argument";
        case FOCUS_ERR_UNSUPPORTED: return "unsupported shape, dtype or alignment";
        case FOCUS_ERR_CAPACITY: return "ring or window buffer capacity exceeded";
        case FOCUS_ERR_CUDA: return "CUDA error";
        case FOCUS_ERR_TIMEOUT: return "bounded device wait timed out";
        case FOCUS_ERR_LAYOUT: return "device layout disagrees with the given sizes";
    }
    return "unknown status";
}

focus_status focus_get_device_status(int32_t* host_status, int32_t clear, cudaStream_t stream) {
    if (!host_status) return FOCUS_ERR_INVALID_ARG;
    int32_t* p = nullptr;
    focus_status st = status_ptr(&p);
    if (st != FOCUS_OK) return st;
    if (cudaStreamSynchronize(stream) != cudaSuccess) return FOCUS_ERR_CUDA;
    if (cudaMemcpy(host_status, p, sizeof(int32_t), cudaMemcpyDeviceToHost) != cudaSuccess) return FOCUS_ERR_CUDA;
    if (clear) {
        if (cudaMemsetAsync(p, 0, sizeof(int32_t), stream) != cudaSuccess) return FOCUS_ERR_CUDA;
        if (cudaStreamSynchronize(stream) != cudaSuccess) return FOCUS_ERR_CUDA;
    }
    return FOCUS_OK;
}

}  // extern "C"

namespace {

// Host sizes of a layout; sched = false means windows of W bases (h_W unused).
focus_status layout_size_impl(int64_t n_nt, int32_t W, bool sched, const int32_t* h_W, int32_t n_windows,
                              const int32_t* h_k, uint32_t flags, int32_t tail, int64_t* T, int64_t* R,
                              int32_t* max_rows) {
    if (n_nt < 0 || tail < 0 || n_windows < 0 || (n_nt > 0 && !h_k)) return FOCUS_ERR_INVALID_ARG;
    if (!sched && (W <= 0 || (int64_t)n_windows != focus::ceil_div64(n_nt, W))) return FOCUS_ERR_INVALID_ARG;
    if (sched && n_windows > 0 && !h_W) return FOCUS_ERR_INVALID_ARG;
    const bool close_tail = (flags & FOCUS_LAYOUT_CLOSE_TAIL) != 0;
    int64_t t = 0, r = 0, mx = 0, start = 0;
    for (int32_t w = 0; w < n_windows; ++w) {
        const int64_t len = sched ? h_W[w] : W;
        if (h_k[w] < 0 || len <= 0 || start >= n_nt) return FOCUS_ERR_INVALID_ARG;
        int64_t n = n_nt - start;
        if (n > len) n = len;
        const int64_t rows = focus::window_rows(n, h_k[w], (w < n_windows - 1) || close_tail);
        t += rows;
        r += rows - n + (n - focus::tail_start(n, tail));
        if (rows > mx) mx = rows;
        start += len;
    }
    if (start < n_nt) return FOCUS_ERR_INVALID_ARG;   // the windows do not cover the sequence
    if (t > INT32_MAX) return FOCUS_ERR_UNSUPPORTED;   // offsets are int32
    if (T) *T = t;
    if (R) *R = r;
    if (max_rows) *max_rows = (int32_t)mx;
    return FOCUS_OK;
}

focus_status layout_impl(int64_t n_nt, int32_t W, bool sched, const int32_t* d_W, int32_t n_windows,
                         const int32_t* d_k, uint32_t flags, int32_t tail, int32_t B, const uint8_t* d_nt,
                         const focus_layout_out* out, cudaStream_t stream) {
    if (!out || n_nt < 0 || B < 0 || tail < 0 || n_windows < 0) return FOCUS_ERR_INVALID_ARG;
    if (!sched && (W <= 0 || (int64_t)n_windows != focus::ceil_div64(n_nt, W))) return FOCUS_ERR_INVALID_ARG;
    if (sched && n_windows > 0 && !d_W) return FOCUS_ERR_INVALID_ARG;
    if (n_nt == 0) {                                   // empty sequence: nothing to lay out
        if (n_windows != 0 || out->T != 0 || out->R != 0) return FOCUS_ERR_INVALID_ARG;
        if (!out->win_off || !out->ring_off) return FOCUS_ERR_INVALID_ARG;
        cudaError_t e = cudaMemsetAsync(out->win_off, 0, sizeof(int32_t), stream);
        if (e == cudaSuccess) e = cudaMemsetAsync(out->ring_off, 0, sizeof(int32_t), stream);
        if (e == cudaSuccess && out->base_off) e = cudaMemsetAsync(out->base_off, 0, sizeof(int32_t), stream);
        return from_cuda(e);
    }
    if (!d_k || n_windows == 0) return FOCUS_ERR_INVALID_ARG;
    if (out->T < 0 || out->R < 0 || out->T > INT32_MAX) return FOCUS_ERR_INVALID_ARG;
    if (!out->win_off || !out->ring_off) return FOCUS_ERR_INVALID_ARG;
    if (sched && !out->base_off) return FOCUS_ERR_INVALID_ARG;
    if (out->T > 0 && (!out->kind || !out->src || !out->pos || !out->win)) return FOCUS_ERR_INVALID_ARG;
    if (out->R > 0 && !out->sum_idx) return FOCUS_ERR_INVALID_ARG;
    if (out->tok && (!d_nt || B <= 0)) return FOCUS_ERR_INVALID_ARG;
    int32_t* st = nullptr;
    focus_status s = status_ptr(&st);
    if (s != FOCUS_OK) return s;
    return from_cuda(focus::launch_layout(n_nt, W, sched ? d_W : nullptr, n_windows, d_k, (flags & FOCUS_LAYOUT_CLOSE_TAIL) != 0, tail,
                                          B, d_nt, *out, st, stream));
}

}  // namespace

extern "C" {

focus_status focus_layout_windows(int64_t n_nt, int32_t W, int32_t* M) {
    if (!M || n_nt < 0 || W < 1) return FOCUS_ERR_INVALID_ARG;
    const int64_t m = focus::ceil_div64(n_nt, W);
    if (m > INT32_MAX) return FOCUS_ERR_INVALID_ARG;
    *M = (int32_t)m;
    return FOCUS_OK;
}

focus_status focus_layout_windows_sched(int64_t n_nt, int32_t n_sched, const int32_t* h_W, int32_t* M) {
    if (!M || n_nt < 0 || n_sched < 0 || (n_sched > 0 && !h_W)) return FOCUS_ERR_INVALID_ARG;
    int64_t covered = 0;
    int32_t m = 0;
    while (covered < n_nt) {
        if (m >= n_sched || h_W[m] < 1) return FOCUS_ERR_INVALID_ARG;
        covered += h_W[m++];
    }
    *M = m;
    return FOCUS_OK;
}

focus_status focus_layout_size(int64_t n_nt, int32_t W, int32_t n_windows, const int32_t* h_k, uint32_t flags,
                               int32_t tail, int64_t* T, int64_t* R, int32_t* max_rows) {
    return layout_size_impl(n_nt, W, false, nullptr, n_windows, h_k, flags, tail, T, R, max_rows);
}

focus_status focus_layout_size_sched(int64_t n_nt, int32_t n_windows, const int32_t* h_W, const int32_t* h_k,
                                     uint32_t flags, int32_t tail, int64_t* T, int64_t* R, int32_t* max_rows) {
    return layout_size_impl(n_nt, 0, true, h_W, n_windows, h_k, flags, tail, T, R, max_rows);
}

focus_status focus_layout(int64_t n_nt, int32_t W, int32_t n_windows, const int32_t* d_k, uint32_t flags,
                          int32_t tail, int32_t B, const uint8_t* d_nt, const focus_layout_out* out,
                          cudaStream_t stream) {
    return layout_impl(n_nt, W, false, nullptr, n_windows, d_k, flags, tail, B, d_nt, out, stream);
}

focus_status focus_layout_sched(int64_t n_nt, int32_t n_windows, const int32_t* d_W, const int32_t* d_k,
                                uint32_t flags, int32_t tail, int32_t B, const uint8_t* d_nt,
                                const focus_layout_out* out, cudaStream_t stream) {
    return layout_impl(n_nt, 0, true, d_W, n_windows, d_k, flags, tail, B, d_nt, out, stream);
}

static focus_status check_prefill(const focus_cache* cache, const focus_prefill_args* a) {
    focus_status s = check_cache(cache, false);
    if (s != FOCUS_OK) return s;
    if (!a || !a->q || !a->k || !a->v || !a->o || !a->d_win_off || !a->d_ring_off) return FOCUS_ERR_INVALID_ARG;
    if (a->w_begin < 0 || a->w_end <= a->w_begin || a->w_end > a->n_windows || a->T_span < 0 || a->max_rows <= 0)
        return FOCUS_ERR_INVALID_ARG;
    if (!isfinite(a->scale) || !(a->scale > 0.f)) return FOCUS_ERR_INVALID_ARG;
    if (!aligned16(a->q) || !aligned16(a->k) || !aligned16(a->v) || !aligned16(a->o)) return FOCUS_ERR_UNSUPPORTED;
    if (a->workspace && !aligned16(a->workspace)) return FOCUS_ERR_UNSUPPORTED;
    if (a->flags & ~(uint32_t)(FOCUS_PREFILL_LEGACY_MMA | FOCUS_PREFILL_KMER_LOCAL)) return FOCUS_ERR_INVALID_ARG;
    if ((a->flags & FOCUS_PREFILL_LEGACY_MMA) && (cache->rope_theta > 0.f || cache->q_per_kv > 1))
        return FOCUS_ERR_UNSUPPORTED;
    if (a->flags & FOCUS_PREFILL_KMER_LOCAL) {
        if (a->flags & FOCUS_PREFILL_LEGACY_MMA) return FOCUS_ERR_UNSUPPORTED;
        if (cache->tail != 0) return FOCUS_ERR_UNSUPPORTED;
        if (!cache->k_per_window || cache->n_windows < a->w_end) return FOCUS_ERR_INVALID_ARG;
    }
    return FOCUS_OK;
}

focus_status focus_prefill_kernel(const focus_cache* cache, const focus_prefill_args* a, int32_t* kernel) {
    if (!kernel) return FOCUS_ERR_INVALID_ARG;
    focus_status s = check_prefill(cache, a);
    if (s != FOCUS_OK) return s;
    *kernel = focus::prefill_kernel_choice(*cache, *a);
    return FOCUS_OK;
}

size_t focus_prefill_workspace_size(const focus_cache* cache, const focus_prefill_args* a) {
    if (check_prefill(cache, a) != FOCUS_OK) return 0;
    return focus::prefill_workspace_bytes(*cache, *a);
}

focus_status focus_attn_prefill(const focus_cache* cache, const focus_prefill_args* a, cudaStream_t stream) {
    focus_status s = check_prefill(cache, a);
    if (s != FOCUS_OK) return s;
    if (a->T_span == 0) return FOCUS_OK;
    const int64_t tiles = focus::ceil_div64(a->max_rows, 64) * (int64_t)(a->w_end - a->w_begin);
    if (tiles > INT32_MAX) return FOCUS_ERR_UNSUPPORTED;
    int32_t* st = nullptr;
    s = status_ptr(&st);
    if (s != FOCUS_OK) return s;
    if (a->flags & FOCUS_PREFILL_LEGACY_MMA) return from_cuda(focus::launch_prefill_mma(*cache, *a, st, stream));
    return from_cuda(focus::launch_prefill_tc(*cache, *a, st, stream));
}

size_t focus_decode_workspace_size(const focus_cache* cache) {
    if (check_cache(cache, false) != FOCUS_OK) return 0;
    return focus::decode_workspace_bytes(*cache);
}

focus_status focus_attn_decode(const focus_cache* cache, const void* q, const void* k_new, const void* v_new,
                               float scale, void* o, float* lse, void* workspace, size_t workspace_bytes,
                               cudaStream_t stream) {
    focus_status s = check_cache(cache, true);
    if (s != FOCUS_OK) return s;
    if (!q || !k_new || !v_new || !o || !workspace || !isfinite(scale)) return FOCUS_ERR_INVALID_ARG;
    if (cache->rope_theta > 0.f && !cache->pos_base) return FOCUS_ERR_INVALID_ARG;
    if (!aligned16(q) || !aligned16(k_new) || !aligned16(v_new) || !aligned16(o) || !aligned16(workspace))
        return FOCUS_ERR_UNSUPPORTED;
    if (workspace_bytes < focus_decode_workspace_size(cache)) return FOCUS_ERR_CAPACITY;
    if (cache->C_ring > 0 && (!cache->ring_k || !cache->ring_v)) return FOCUS_ERR_INVALID_ARG;
    int32_t* st = nullptr;
    s = status_ptr(&st);
    if (s != FOCUS_OK) return s;
    return from_cuda(focus::launch_decode(*cache, q, k_new, v_new, scale, o, lse, workspace, st, stream));
}

focus_status focus_attn_decode_noalloc(const focus_cache* cache, const void* q, const void* k_new,
                                       const void* v_new, float scale, void* o, float* lse, cudaStream_t stream) {
    focus_status s = check_cache(cache, true);
    if (s != FOCUS_OK) return s;
    if (!q || !k_new || !v_new || !o || !isfinite(scale)) return FOCUS_ERR_INVALID_ARG;
    if (cache->rope_theta > 0.f && !cache->pos_base) return FOCUS_ERR_INVALID_ARG;
    if (!aligned16(q) || !aligned16(k_new) || !aligned16(v_new) || !aligned16(o)) return FOCUS_ERR_UNSUPPORTED;
    if (focus_decode_workspace_size(cache) > (size_t)FOCUS_DECODE_NOALLOC_SCRATCH_BYTES) return FOCUS_ERR_CAPACITY;
    int32_t* st = nullptr;
    s = status_ptr(&st);
    if (s != FOCUS_OK) return s;
    return from_cuda(focus::launch_decode_noalloc(*cache, q, k_new, v_new, scale, o, lse, st, stream));
}

focus_status focus_kv_compact(const focus_cache* cache, const focus_compact_args* a, cudaStream_t stream) {
    if (!a) return FOCUS_ERR_INVALID_ARG;
    const bool bulk = a->src_k != nullptr;
    focus_status s = check_cache(cache, !bulk);
    if (s != FOCUS_OK) return s;
    if (!cache->ring_k || !cache->ring_v || !cache->ring_len) return FOCUS_ERR_INVALID_ARG;
    int32_t* st = nullptr;
    s = status_ptr(&st);
    if (s != FOCUS_OK) return s;
    if (bulk) {
        if (!a->src_v || !a->d_sum_idx || !a->d_ring_off || a->src_T < 0 || a->w_begin < 0 || a->w_end < a->w_begin ||
            a->w_end > a->n_windows)
            return FOCUS_ERR_INVALID_ARG;
        if (!aligned16(a->src_k) || !aligned16(a->src_v)) return FOCUS_ERR_UNSUPPORTED;
        if (a->w_end == a->w_begin) return FOCUS_OK;
        if (cache->rope_theta > 0.f) return from_cuda(focus::launch_compact_bulk_rope(*cache, *a, st, stream));
        return from_cuda(focus::launch_compact_bulk(*cache, *a, st, stream));
    }
    return from_cuda(focus::launch_compact_window(*cache, st, stream));
}

focus_status focus_selftest_timeout(uint64_t limit_ns, cudaStream_t stream) {
    if (limit_ns == 0 || limit_ns > 10000000000ull) return FOCUS_ERR_INVALID_ARG;
    int32_t* st = nullptr;
    focus_status s = status_ptr(&st);
    if (s != FOCUS_OK) return s;
    return from_cuda(focus::launch_selftest_timeout(limit_ns, st, stream));
}

focus_status focus_embed_tokens(const uint8_t* d_tok, int64_t n_rows, const void* d_table, int32_t n_tokens,
                                int32_t D, void* d_out, cudaStream_t stream) {
    if (n_rows < 0 || n_tokens < 1 || n_tokens > 256 || D <= 0) return FOCUS_ERR_INVALID_ARG;
    if (D % 8 != 0) return FOCUS_ERR_UNSUPPORTED;
    if (n_rows == 0) return FOCUS_OK;
    if (!d_tok || !d_table || !d_out) return FOCUS_ERR_INVALID_ARG;
    if (!aligned16(d_table) || !aligned16(d_out)) return FOCUS_ERR_UNSUPPORTED;
    if (n_rows > INT64_MAX / D) return FOCUS_ERR_UNSUPPORTED;
    int32_t* st = nullptr;
    focus_status s = status_ptr(&st);
    if (s != FOCUS_OK) return s;
    return from_cuda(focus::launch_embed_tokens(d_tok, n_rows, d_table, n_tokens, D, d_out, st, stream));
}

}  // extern "C"
